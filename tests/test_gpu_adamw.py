"""GPU parity of the fused AdamW step (UF8 momentum, AL-coded V) with the
oracle.

Sec. 3.1 Eq. (1), Sec. 6.2, Sec. 7.1. Both sides run the same steps from the
same seeded state and gradients; codes and block metadata must agree bit for
bit after every step (the arithmetic contract fixes the fp32 operation order,
and the codec's fast paths fall back to the defining double expressions near
rounding boundaries). Parameters agree within 1e-5 of |p| plus the summed
step sizes: the kernel's update direction takes the approximate square root
and reciprocal, which move p alone. Covered: the 256x1024 single-tensor
workload for 10 steps (persistent and redrawn zero masks), the paper's
B_V = 2048 setting, AL16, every block-size class, ragged lengths, a
multi-tensor plan with tiny and ragged tensors, and the full 1.1B-parameter
TinyLlama plan checked on sampled blocks.
"""
import numpy as np
import pytest

import oracle as ora
from gpu_util import ADAMW_HP, bytes_equal, gpu_available, params_off, step_size
from paper_2608_22322_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not gpu_available(), reason="needs a CUDA GPU")]


@pytest.fixture(scope="module")
def B():
    from paper_2608_22322_gb300 import binding
    return binding


class Pair:
    """The same AdamW state on the host (oracle) and the device (library)."""

    def __init__(self, p0, m_block, v_block, v_bits):
        import torch
        n = p0.size
        self.n, self.mb, self.vb, self.bits = n, m_block, v_block, v_bits
        self.h = dict(p=p0.ravel().copy(), mc=np.zeros(n, np.int8),
                      ma=np.zeros((n + m_block - 1) // m_block, np.float32),
                      vc=np.zeros(n, ora.code_dtype(v_bits)),
                      vm=np.zeros(2 * ((n + v_block - 1) // v_block), np.float32))
        self.steps = np.zeros(n)  # summed |lr u| of the oracle's steps
        self.d = {k: torch.from_numpy(v.view(np.int16) if v.dtype == np.uint16 else v.copy()).cuda()
                  for k, v in self.h.items()}

    def host_step(self, g, t, hp=ADAMW_HP):
        h = self.h
        p_old = h["p"].copy()
        ora.adamw_step(h["p"], g, h["mc"], h["ma"], h["vc"], h["vm"], self.mb, self.vb,
                       self.bits, hp, t)
        self.steps += step_size(h["p"], p_old, hp)

    def dev_args(self):
        d = self.d
        return dict(p=d["p"], m_codes=d["mc"], m_absmax=d["ma"], v_codes=d["vc"], v_meta=d["vm"])

    def compare(self, what=""):
        import torch
        torch.cuda.synchronize()
        for k in ("p", "mc", "ma", "vc", "vm"):
            got = self.d[k].cpu().numpy()
            if k == "p":
                bad = params_off(self.h[k], got, self.steps)
                assert bad == 0, f"{what}: {bad} parameters outside the tolerance"
            else:
                bad = bytes_equal(self.h[k], got)
                assert bad == 0, f"{what}: {k} differs in {bad} bytes"


def _run_single(B, w, m_block, v_block, v_bits, steps, hp=ADAMW_HP):
    import torch
    pr = Pair(w.p0, m_block, v_block, v_bits)
    for t in range(1, steps + 1):
        g = w.grad(t).ravel()
        pr.host_step(g, t, hp)
        a = pr.dev_args()
        B.al_adamw_step(a["p"], torch.from_numpy(g).cuda(), a["m_codes"], a["m_absmax"],
                        a["v_codes"], a["v_meta"], m_block, v_block, v_bits, hp, t)
        pr.compare(f"step {t}")
    return pr


def test_adamw_256x1024_ten_steps(B):
    """The single-tensor workload: 256x1024, 10% zero mask, 2% dormant rows,
    AL8/UF8 blocks of 256, wd 0.01, 10 steps."""
    w = wl.AdamWSingle()
    pr = _run_single(B, w, 256, 256, 8, 10)
    codes = pr.h["vc"].reshape(w.shape)
    assert not codes[w.dormant].any()


def test_adamw_redrawn_mask(B):
    w = wl.AdamWSingle(redraw_mask=True)
    _run_single(B, w, 256, 256, 8, 5)


@pytest.mark.parametrize("m_block,v_block", [(256, 2048), (128, 128), (512, 1024),
                                             (2048, 256), (128, 2048), (128, 256),
                                             (256, 128), (2048, 128), (512, 512),
                                             (256, 4096), (4096, 128), (4096, 4096)])
def test_adamw_block_sizes(B, m_block, v_block):
    w = wl.AdamWSingle(shape=(37, 1111))  # 41107 elements: ragged tiles and blocks
    _run_single(B, w, m_block, v_block, 8, 4)


@pytest.mark.parametrize("m_block,v_block", [(256, 256), (256, 128), (128, 1024)])
def test_adamw_al16(B, m_block, v_block):
    w = wl.AdamWSingle(shape=(64, 777))
    _run_single(B, w, m_block, v_block, 16, 4)


@pytest.mark.parametrize("v_block", [2048, 256])
def test_adamw_plan_many_tensors(B, v_block):
    """Multi-tensor plan: tiny, ragged and multi-tile tensors in one launch
    (V blocks of 2048 shared by a CTA's warps; of 256, one per warp with
    the warp pairs' shared level pass)."""
    import torch
    sizes = [1, 5, 4095, 4097, 300, 2 * 4096 + 511, 17, 64 * 1024]
    pairs, gens = [], []
    for i, n in enumerate(sizes):
        p0 = wl.param_init((n,), 40 + i, norm_vector_value=0.5) if i % 2 else \
            (wl.rng(40 + i).standard_normal(n) * 0.02).astype(np.float32)
        pairs.append(Pair(p0, 256, v_block, 8))
        gens.append(lambda t, n=n, i=i: wl.gaussian_grad((n,), 1e-3, 900 + 31 * i + t,
                                                         wl.zero_mask((n,), 0.1, 77 + i)))
    gdev = [torch.zeros(n, dtype=torch.float32, device="cuda") for n in sizes]
    plan = B.AdamWPlan([dict(g=gdev[i], **pr.dev_args()) for i, pr in enumerate(pairs)],
                       256, v_block, 8)
    for t in range(1, 4):
        for i, pr in enumerate(pairs):
            g = gens[i](t)
            pr.host_step(g, t)
            gdev[i].copy_(torch.from_numpy(g))
        plan.step(ADAMW_HP, t)
        for i, pr in enumerate(pairs):
            pr.compare(f"tensor {i} (n={sizes[i]}) step {t}")


def test_adamw_plan_over_pinned_host_buffers(B):
    """A plan whose parameters, gradients, codes and block constants are
    pinned host memory (their device mapping): the kernel steps them in
    place across the host link, as the end-to-end bench does, with the same
    results as on device buffers (the oracle's, bit for bit for codes and
    constants)."""
    import torch
    sizes = [5, 4097, 2 * 4096 + 511, 64 * 1024]
    pairs, gens = [], []
    for i, n in enumerate(sizes):
        p0 = (wl.rng(60 + i).standard_normal(n) * 0.02).astype(np.float32)
        pr = Pair(p0, 256, 256, 8)
        pr.d = {k: v.cpu().pin_memory() for k, v in pr.d.items()}
        pairs.append(pr)
        gens.append(lambda t, n=n, i=i: wl.gaussian_grad((n,), 1e-3, 700 + 31 * i + t,
                                                         wl.zero_mask((n,), 0.1, 57 + i)))
    ghost = [torch.zeros(n, dtype=torch.float32).pin_memory() for n in sizes]
    plan = B.AdamWPlan([dict(g=ghost[i], **pr.dev_args()) for i, pr in enumerate(pairs)],
                       256, 256, 8, device=torch.device("cuda"))
    for t in range(1, 4):
        torch.cuda.synchronize()
        for i, pr in enumerate(pairs):
            g = gens[i](t)
            pr.host_step(g, t)
            ghost[i].copy_(torch.from_numpy(g))
        plan.step(ADAMW_HP, t)
        for i, pr in enumerate(pairs):
            pr.compare(f"host tensor {i} (n={sizes[i]}) step {t}")


def test_adamw_tinyllama_full_plan_sampled(B):
    """All 201 TinyLlama-1.1B tensors (1,100,048,384 parameters) in one plan,
    the launch the benchmark times. Blocks are independent in AdamW, so the
    oracle re-runs sampled blocks (first, last and random ones of every tensor)
    from a snapshot of their state and gradient, step by step."""
    import torch
    cfg = wl.CONFIGS["tinyllama_adamw"]
    mb, vb = cfg["m_block"], cfg["v_block"]
    tens = wl.tinyllama_tensors()
    dev = []
    for i, (name, shape) in enumerate(tens):
        n = wl.numel(shape)
        p = torch.empty(n, dtype=torch.float32, device="cuda")
        if len(shape) == 1:
            p.fill_(1.0)
        else:
            wl.torch_device_normal_(p, 0.02, 1000 + i)
        dev.append(dict(p=p, g=torch.empty(n, dtype=torch.float32, device="cuda"),
                        m_codes=torch.zeros(n, dtype=torch.int8, device="cuda"),
                        m_absmax=torch.zeros((n + mb - 1) // mb, dtype=torch.float32, device="cuda"),
                        v_codes=torch.zeros(n, dtype=torch.uint8, device="cuda"),
                        v_meta=torch.zeros(2 * ((n + vb - 1) // vb), dtype=torch.float32,
                                           device="cuda")))
    plan = B.AdamWPlan(dev, mb, vb, 8)
    assert plan.info.total_elems == 1_100_048_384
    r = wl.rng(5)
    samples = []
    for i, (_, shape) in enumerate(tens):
        nb = (wl.numel(shape) + 255) // 256
        picks = {0, nb - 1, *map(int, r.integers(0, nb, 2))}
        samples += [(i, b) for b in sorted(picks)]
    for t in (1, 2, 3):
        for i, d in enumerate(dev):
            wl.torch_device_normal_(d["g"], 1e-3, 50_000 + 1000 * t + i)
            wl.torch_device_zero_(d["g"], 0.01, 90_000 + 1000 * t + i)
        snap = []
        for i, b in samples:
            d = dev[i]
            lo, hi = 256 * b, min(256 * (b + 1), d["p"].numel())
            snap.append(dict(p=d["p"][lo:hi].cpu().numpy(), g=d["g"][lo:hi].cpu().numpy(),
                             mc=d["m_codes"][lo:hi].cpu().numpy(),
                             ma=d["m_absmax"][b:b + 1].cpu().numpy(),
                             vc=d["v_codes"][lo:hi].cpu().numpy(),
                             vm=d["v_meta"][2 * b:2 * b + 2].cpu().numpy()))
        plan.step(ADAMW_HP, t)
        torch.cuda.synchronize()
        for (i, b), s in zip(samples, snap):
            p_old = s["p"].copy()
            ora.adamw_step(s["p"], s["g"], s["mc"], s["ma"], s["vc"], s["vm"], 256, 256, 8,
                           ADAMW_HP, t)
            d = dev[i]
            lo, hi = 256 * b, min(256 * (b + 1), d["p"].numel())
            assert params_off(s["p"], d["p"][lo:hi].cpu().numpy(),
                              step_size(s["p"], p_old, ADAMW_HP)) == 0, (tens[i][0], b, t)
            for k, got in (("mc", d["m_codes"][lo:hi]),
                           ("ma", d["m_absmax"][b:b + 1]), ("vc", d["v_codes"][lo:hi]),
                           ("vm", d["v_meta"][2 * b:2 * b + 2])):
                assert bytes_equal(s[k], got.cpu().numpy()) == 0, (tens[i][0], b, k, t)
    del dev, plan
    torch.cuda.empty_cache()


def test_adamw_rejects_bad_arguments(B):
    import torch
    x = torch.zeros(1024, device="cuda")
    c = torch.zeros(1024, dtype=torch.int8, device="cuda")
    with pytest.raises(B.AlqError, match="UNSUPPORTED"):
        B.al_adamw_step(x, x, c, x, c, x, 100, 256, 8, ADAMW_HP, 1)
    with pytest.raises(B.AlqError, match="ALIGN"):
        B.al_adamw_step(x[1:], x[1:], c[1:], x, c[1:], x, 256, 256, 8, ADAMW_HP, 1)
    with pytest.raises(B.AlqError, match="INVALID_ARG"):
        B.al_adamw_step(x, x, c, x, c, x, 256, 256, 8, ADAMW_HP, 0)


def test_adamw_fp32_role_single_and_plan(B):
    """v_bits = 32 (dense fp32 m and v, Sec. 4.5's FP32 role): the kernel's
    parameters and states equal the oracle's bit for bit, single tensor and
    multi-tensor plan, ragged sizes."""
    import torch
    sizes = [41107, 5, 4096 * 3 + 17]
    hs, ds, gds = [], [], []
    for i, n in enumerate(sizes):
        p0 = (wl.rng(500 + i).standard_normal(n) * 0.02).astype(np.float32)
        h = dict(p=p0.copy(), m=np.zeros(n, np.float32), v=np.zeros(n, np.float32))
        hs.append(h)
        ds.append({k: torch.from_numpy(v.copy()).cuda() for k, v in h.items()})
        gds.append(torch.zeros(n, dtype=torch.float32, device="cuda"))
    plan = B.AdamWPlan([dict(p=d["p"], g=g, m_codes=d["m"], m_absmax=None, v_codes=d["v"],
                             v_meta=None) for d, g in zip(ds[1:], gds[1:])], 256, 256, 32)
    for t in range(1, 5):
        for i, n in enumerate(sizes):
            g = wl.gaussian_grad((n,), 1e-3, 600 + 10 * t + i, wl.zero_mask((n,), 0.05, 7 + i))
            h = hs[i]
            ora.adamw_step(h["p"], g, h["m"], None, h["v"], None, 256, 256, 32, ADAMW_HP, t)
            gds[i].copy_(torch.from_numpy(g))
        B.al_adamw_step(ds[0]["p"], gds[0], ds[0]["m"], None, ds[0]["v"], None, 256, 256, 32,
                        ADAMW_HP, t)
        plan.step(ADAMW_HP, t)
        torch.cuda.synchronize()
        for h, d in zip(hs, ds):
            for k in ("p", "m", "v"):
                assert bytes_equal(h[k], d[k].cpu().numpy()) == 0, (t, k, h["p"].size)


def test_adamw_beyond_2_31_elements_sampled(B):
    """One tensor of 2^31 + 4099 parameters (64-bit indexing in the kernel):
    sampled blocks below and above 2^31, and the ragged last block, against
    the oracle re-run from a snapshot of each block (blocks are independent).
    An empty tensor next to it in a plan is a no-op."""
    import torch
    n = (1 << 31) + 4099
    nb = (n + 255) // 256
    p = torch.empty(n, dtype=torch.float32, device="cuda")
    wl.torch_device_normal_(p, 0.02, 77)
    g = torch.empty(n, dtype=torch.float32, device="cuda")
    d = dict(p=p, g=g, m_codes=torch.zeros(n, dtype=torch.int8, device="cuda"),
             m_absmax=torch.zeros(nb, dtype=torch.float32, device="cuda"),
             v_codes=torch.zeros(n, dtype=torch.uint8, device="cuda"),
             v_meta=torch.zeros(2 * nb, dtype=torch.float32, device="cuda"))
    e = {k: torch.zeros(0, dtype=v.dtype, device="cuda") for k, v in d.items()}
    plan = B.AdamWPlan([e, d], 256, 256, 8)
    assert plan.info.total_elems == n
    picks = [0, 3, (1 << 23) - 1, 1 << 23, (1 << 23) + 1, nb - 2, nb - 1]
    for t in (1, 2):
        wl.torch_device_normal_(g, 1e-3, 500 + t)
        wl.torch_device_zero_(g, 0.01, 600 + t)
        snap = []
        for b in picks:
            lo, hi = 256 * b, min(256 * (b + 1), n)
            snap.append(dict(p=p[lo:hi].cpu().numpy(), g=g[lo:hi].cpu().numpy(),
                             mc=d["m_codes"][lo:hi].cpu().numpy(),
                             ma=d["m_absmax"][b:b + 1].cpu().numpy(),
                             vc=d["v_codes"][lo:hi].cpu().numpy(),
                             vm=d["v_meta"][2 * b:2 * b + 2].cpu().numpy()))
        plan.step(ADAMW_HP, t)
        torch.cuda.synchronize()
        for b, s in zip(picks, snap):
            p_old = s["p"].copy()
            ora.adamw_step(s["p"], s["g"], s["mc"], s["ma"], s["vc"], s["vm"], 256, 256, 8,
                           ADAMW_HP, t)
            lo, hi = 256 * b, min(256 * (b + 1), n)
            assert params_off(s["p"], p[lo:hi].cpu().numpy(),
                              step_size(s["p"], p_old, ADAMW_HP)) == 0, (b, t)
            for k, got in (("mc", d["m_codes"][lo:hi]),
                           ("ma", d["m_absmax"][b:b + 1]), ("vc", d["v_codes"][lo:hi]),
                           ("vm", d["v_meta"][2 * b:2 * b + 2])):
                assert bytes_equal(s[k], got.cpu().numpy()) == 0, (b, k, t)
    assert (nb - 1) * 256 > (1 << 31) and n - (nb - 1) * 256 == 3  # ragged last block
    del d, p, g, plan
    torch.cuda.empty_cache()


def test_adamw_empty_tensor_is_a_noop(B):
    import torch
    z = torch.zeros(0, device="cuda")
    zc = torch.zeros(0, dtype=torch.int8, device="cuda")
    B.al_adamw_step(z, z, zc, z, zc, z, 256, 256, 8, ADAMW_HP, 1)
    torch.cuda.synchronize()
