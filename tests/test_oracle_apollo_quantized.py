"""Pins of the oracle's quantized APOLLO step (Sec. 3.1 APOLLO with the
codecs of Sec. 4.1 Eq. (3)-(5) and Sec. 4.3), of Eq. (2)'s relative update
error, and of the oracle's bf16 rounding.

The fp32-state APOLLO update is pinned elsewhere (torch Adam on an identity
projection, an orthogonal projection's closed form, transpose symmetry, the
limiter's bound). Here the quantized step is pinned by what the paper fixes
about its states and by independent references:
  * hand-built projected states: with an identity projection R is known
    exactly, so the fresh fp32 states at t = 1 and t = 2 follow from the EMA
    definitions; the V^P codes and block constants must be those of the AL
    codec over blocks of one channel (block = rank) with the given floor,
    and the M^P codes those of UF8 with its own block size;
  * dormant channels (an all-zero gradient column or row) keep zero codes,
    a zero channel scale and a parameter that only decays (Eq. (6));
  * tracking: against the fp32-state step whose momentum goes through the
    same UF8 round trip, the displacement error (Eq. (2)) is the second
    moment's quantization error alone -- AL8 within a few 1e-4, AL16 two
    orders of magnitude closer -- and the momentum codes agree exactly, for
    both orientations of the projection.
"""
import math

import numpy as np
import pytest
import torch

import oracle as ora
from paper_2608_22322_gb300 import workloads as wl

FLOOR = float(np.float32(math.log2(1e-16)))
HP = dict(lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, alpha=1.0,
          weight_decay=0.0, norm_growth_gamma=0.0, log_floor=FLOOR)
F32 = np.float32


def _bf16_exact(x):
    return (wl.bf16_bits(x).astype(np.uint32) << 16).view(np.float32)


def _states(L, rank, m_block, v_bits):
    npj = L * rank
    return (np.zeros(npj, np.int8), np.zeros(-(-npj // m_block), np.float32),
            np.zeros(npj, ora.code_dtype(v_bits)), np.zeros(2 * L, np.float32))


# ------------------------------------------------- hand-built projected states
@pytest.mark.parametrize("v_bits", [8, 16])
def test_projected_states_are_coded_per_channel(v_bits):
    """P = I (rank = rows = 8, exact in bf16) and a bf16-exact G: R[j] is
    column j of G. Channel 3 lies below the floor (its V^P block clamps
    l_min to the floor), channel 5 is all zero (no positive value: codes 0,
    constants (0, 0)), the others span nine decades, so a block spanning two
    channels would get other constants. M^P is coded in blocks of 16 (two
    channels), V^P in blocks of rank."""
    rows, cols, rank, m_block = 8, 24, 8, 16
    hp = dict(HP, rank=rank)
    P = wl.bf16_bits(np.eye(rows, dtype=np.float32))
    r = wl.rng(31)

    def grad(seed_shift):
        scale = 10.0 ** r.uniform(-6, 3, size=(1, cols))
        G = r.standard_normal((rows, cols)) * scale
        G[:, 3] = 1e-9 * r.standard_normal(rows)  # (1 - b2) R^2 < 2^floor
        G[:, 5] = 0.0
        return _bf16_exact(G.astype(np.float32))

    mc, ma, vc, vm = _states(cols, rank, m_block, v_bits)
    b1, b2 = F32(hp["beta1"]), F32(hp["beta2"])
    # 1 - beta in double from the fp32 hyperparameter, rounded once
    omb1, omb2 = F32(1.0 - float(b1)), F32(1.0 - float(b2))
    p = np.zeros(rows * cols, np.float32)
    mp_dec = np.zeros(cols * rank, np.float32)
    vp_dec = np.zeros(cols * rank, np.float32)
    for t in (1, 2):
        G = grad(t)
        R = np.ascontiguousarray(G.T).ravel()  # channel-major [cols][rank]
        _, _, MPf, VPf = ora.apollo_step(p, G.ravel(), rows, cols, P, mc, ma, m_block, vc, vm,
                                         v_bits, rank, 0.0, hp, t, want_fresh=True)
        # the EMAs of Sec. 3.1 from the decoded previous states
        want_m = b1 * mp_dec + omb1 * R
        want_v = b2 * vp_dec + omb2 * (R * R)
        np.testing.assert_array_equal(MPf.view(np.uint32), want_m.view(np.uint32))
        np.testing.assert_array_equal(VPf.view(np.uint32), want_v.view(np.uint32))
        # V^P coded per channel (block = rank) with the floor; M^P per m_block
        want_vc, want_vm = ora.al_encode(want_v, rank, v_bits, FLOOR)
        want_mc, want_ma = ora.uf8_encode(want_m, m_block)
        np.testing.assert_array_equal(vc, want_vc)
        np.testing.assert_array_equal(vm.view(np.uint32), want_vm.view(np.uint32))
        np.testing.assert_array_equal(mc, want_mc)
        np.testing.assert_array_equal(ma.view(np.uint32), want_ma.view(np.uint32))
        meta = vm.reshape(cols, 2)
        assert meta[3, 0] == F32(FLOOR)              # below the floor: clamped
        assert tuple(meta[5]) == (0.0, 0.0)          # dormant channel
        assert np.all(vc.reshape(cols, rank)[5] == 0) and np.all(mc.reshape(cols, rank)[5] == 0)
        assert len(set(meta[:, 0].tolist())) >= cols - 2  # one l_min per channel
        # the next step decodes what was stored
        mp_dec = ora.uf8_decode(mc, ma, m_block)
        vp_dec = ora.al_decode(vc, vm, rank, v_bits)


# ---------------------------------------------------------- dormant channels
@pytest.mark.parametrize("shape", [(16, 48), (48, 16)])
def test_dormant_channels_keep_zero_codes_and_only_decay(shape):
    """An all-zero channel of G (a column when rows <= cols, else a row)
    projects to R = 0: its M^P and V^P codes stay 0, its V^P constants
    (0, 0), its scale 0, and its parameters only decay (Eq. (6))."""
    rows, cols = shape
    rank = 8
    hp = dict(HP, rank=rank, weight_decay=0.01)
    short, L = min(shape), max(shape)
    P = wl.bf16_bits(wl.gaussian_projection(rank, short, 12))
    dormant = [2, 7, L - 1]
    mc, ma, vc, vm = _states(L, rank, rank, 8)
    p0 = wl.param_init(shape, 4)
    p = p0.ravel().copy()
    decay = F32(1.0 - 1e-4 * 0.01)
    pd = p0.copy()
    for t in range(1, 6):
        G = wl.gaussian_grad(shape, 1e-3, 40 + t)
        if rows <= cols:
            G[:, dormant] = 0.0
        else:
            G[dormant, :] = 0.0
        s, _ = ora.apollo_step(p, G.ravel(), rows, cols, P, mc, ma, rank, vc, vm, 8, rank, 0.0,
                               hp, t)
        pd = pd * decay
        assert np.all(s[dormant] == 0.0) and np.all(s[[j for j in range(L) if j not in dormant]] > 0)
    for j in dormant:
        assert np.all(mc.reshape(L, rank)[j] == 0) and np.all(vc.reshape(L, rank)[j] == 0)
        assert tuple(vm.reshape(L, 2)[j]) == (0.0, 0.0)
    pm = p.reshape(shape)
    got = pm[:, dormant] if rows <= cols else pm[dormant, :]
    want = pd[:, dormant] if rows <= cols else pd[dormant, :]
    np.testing.assert_array_equal(got, want)


# -------------------------------------------------------------- tracking
def _tracking(rows, cols, rank, v_bits, T=10, seed=0):
    """Displacement and scale errors (Eq. (2)) of the quantized step against
    the fp32-state step whose momentum passes through the same UF8 round
    trip, and whether the momentum codes agree."""
    hp = dict(HP, rank=rank)
    short, L = min(rows, cols), max(rows, cols)
    P = wl.bf16_bits(wl.gaussian_projection(rank, short, 5 + seed))
    p0 = wl.param_init((rows, cols), 3 + seed).ravel()
    p, pf = p0.copy(), p0.copy()
    mc, ma, vc, vm = _states(L, rank, rank, v_bits)
    mc_ref, ma_ref = mc.copy(), ma.copy()
    VP = np.zeros(L * rank, np.float32)
    for t in range(1, T + 1):
        G = wl.gaussian_grad((rows, cols), 1e-3, 100 * seed + t).ravel()
        s, _ = ora.apollo_step(p, G, rows, cols, P, mc, ma, rank, vc, vm, v_bits, rank, 0.0,
                               hp, t)
        MP = ora.uf8_decode(mc_ref, ma_ref, rank)
        sf, _ = ora.apollo_update_fp32(pf, G, rows, cols, P, MP, VP, 0.0, hp, t)
        mc_ref, ma_ref = ora.uf8_encode(MP, rank)
    return (ora.update_error(p - p0, pf - p0), ora.update_error(s, sf),
            np.array_equal(mc, mc_ref))


@pytest.mark.parametrize("shape", [(16, 96), (96, 16), (32, 200)])
def test_quantized_step_tracks_fp32_within_the_codec_error(shape):
    e8, s8, m8 = _tracking(*shape, 16, 8)
    e16, s16, m16 = _tracking(*shape, 16, 16)
    # AL8: half a log-step of Delta / 254 per value, averaged over a channel
    assert 1e-5 < e8 < 3e-3 and s8 < 3e-3, (e8, s8)
    # AL16: 65534 levels instead of 254
    assert e16 < e8 / 30 and s16 < s8 / 30, (e16, e8, s16, s8)
    # the momentum does not depend on the second moment
    assert m8 and m16


def test_given_R_equals_projected_step():
    """The teacher-forced entry point (R given) is the step after the
    projection: fed the oracle's own projection it reproduces apollo_step
    bit for bit."""
    rows, cols, rank = 24, 64, 8
    hp = dict(HP, rank=rank, norm_growth_gamma=1.01)
    P = wl.bf16_bits(wl.gaussian_projection(rank, rows, 9))
    a = [wl.param_init((rows, cols), 1).ravel(), *_states(cols, rank, rank, 8), F32(0.0)]
    b = [x.copy() for x in a]
    for t in range(1, 4):
        G = wl.gaussian_grad((rows, cols), 1e-3, 7 + t).ravel()
        sa, a[5] = ora.apollo_step(a[0], G, rows, cols, P, a[1], a[2], rank, a[3], a[4], 8,
                                   rank, a[5], hp, t)
        R = ora.apollo_project(G, rows, cols, P, rank)
        sb, b[5] = ora.apollo_step_given_R(b[0], G, rows, cols, R, b[1], b[2], rank, b[3],
                                           b[4], 8, rank, b[5], hp, t)
        np.testing.assert_array_equal(sa, sb)
        for x, y in zip(a, b):
            np.testing.assert_array_equal(np.asarray(x), np.asarray(y))


# ------------------------------------------------------------------ Eq. (2)
def test_update_error_closed_forms():
    """Eq. (2), ||u_hat - u|| / (||u|| + eps): a scaled update (1 + d) u
    gives |d|; an orthogonal perturbation gives its norm ratio (3-4-5); a
    zero update gives 1; eps only guards the zero reference."""
    u = wl.rng(3).standard_normal(1000).astype(np.float32)
    for d in (0.25, -0.5, 2.0 ** -10):
        uh = (u.astype(np.float64) * (1.0 + d)).astype(np.float32)
        want = np.linalg.norm(uh.astype(np.float64) - u) / np.linalg.norm(u.astype(np.float64))
        assert abs(ora.update_error(uh, u) - abs(d)) < 1e-6 * abs(d) + 1e-7
        assert abs(ora.update_error(uh, u) - want) < 1e-12
    a = np.array([3.0, 0.0, 0.0], np.float32)
    assert ora.update_error(a + np.array([0.0, 4.0, 0.0], np.float32), a) == pytest.approx(4.0 / 3.0, rel=1e-12)
    assert ora.update_error(np.zeros(3, np.float32), a) == pytest.approx(1.0, rel=1e-12)
    assert ora.update_error(np.zeros(3, np.float32), np.zeros(3, np.float32)) == 0.0
    # the error is not symmetric: the reference's norm is the denominator
    assert ora.update_error(a, 2 * a) == pytest.approx(0.5, rel=1e-12)
    assert ora.update_error(2 * a, a) == pytest.approx(1.0, rel=1e-12)


# -------------------------------------------------------------------- bf16
def test_bf16_rounding_matches_torch():
    """The oracle's fp32 -> bf16 rounding (nearest even) against torch's,
    including exact ties and values at the top of a binade."""
    r = wl.rng(77)
    x = (r.standard_normal(4096) * 10.0 ** r.uniform(-20, 20, 4096)).astype(np.float32)
    base = x.view(np.uint32) & np.uint32(0xFFFF0000)
    ties = (base | np.uint32(0x8000)).view(np.float32)           # exact halfway
    tops = (np.uint32(0x3F7FFFFF) + np.arange(8, dtype=np.uint32) * np.uint32(0x800000)).view(np.float32)
    allx = np.concatenate([x, ties, tops, -ties[:64]])
    got = ora.f32_to_bf16(allx)
    want = torch.from_numpy(allx.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(got, want)
    back = ora.bf16_to_f32(got)
    np.testing.assert_array_equal(back, torch.from_numpy(want.view(np.int16).copy()).view(torch.bfloat16).float().numpy())
