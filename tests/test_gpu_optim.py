"""The torch.optim wrappers (paper_2608_22322_gb300/optim.py) against direct
C-ABI calls: the wrappers only group parameters and keep state, so every
step must equal the direct calls bit for bit. Also covered: torch.optim
conventions (closures, learning-rate schedulers, state_dict round trips with
integer code tensors), AL8 <-> AL16 migration of trained states (Sec. 6.2
per-role precision), and APOLLO's routing of non-matrix parameters to the
quantized AdamW step."""
import math

import numpy as np
import pytest

from gpu_util import ADAMW_HP, gpu_available
from paper_2608_22322_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not gpu_available(), reason="needs a CUDA GPU")]


@pytest.fixture(scope="module")
def mods():
    from paper_2608_22322_gb300 import binding, optim
    return binding, optim


def _params(shapes, seed):
    import torch
    return [torch.nn.Parameter(torch.from_numpy(wl.param_init(s, seed + i)).cuda())
            for i, s in enumerate(shapes)]


def _grads(params, t, seed):
    import torch
    for i, p in enumerate(params):
        p.grad = torch.from_numpy(
            wl.gaussian_grad(tuple(p.shape), 1e-3, seed + 100 * t + i,
                             wl.zero_mask(tuple(p.shape), 0.05, seed + i))).cuda()


def _same(a, b):
    return np.array_equal(a.detach().cpu().numpy().view(np.uint8),
                          b.detach().cpu().numpy().view(np.uint8))


def test_adamw_wrapper_matches_fused_plan(mods):
    """Three parameters, three steps, a scheduler halving lr after step 1:
    the wrapper's parameters and codes equal al_adamw_step_multi's."""
    import torch
    B, optim = mods
    shapes = [(64, 300), (2048,), (37, 111)]
    pw, pd = _params(shapes, 10), _params(shapes, 10)
    opt = optim.AdamW(pw, lr=1e-3, weight_decay=0.01)
    sched = torch.optim.lr_scheduler.StepLR(opt, step_size=1, gamma=0.5)
    st = [dict(m_codes=torch.zeros(p.numel(), dtype=torch.int8, device="cuda"),
               m_absmax=torch.zeros((p.numel() + 255) // 256, dtype=torch.float32, device="cuda"),
               v_codes=torch.zeros(p.numel(), dtype=torch.uint8, device="cuda"),
               v_meta=torch.zeros(2 * ((p.numel() + 255) // 256), dtype=torch.float32,
                                  device="cuda")) for p in pd]
    lr = 1e-3
    for t in (1, 2, 3):
        _grads(pw, t, 500)
        _grads(pd, t, 500)
        opt.step()
        sched.step()
        plan = B.AdamWPlan([dict(p=p.data, g=p.grad, **s) for p, s in zip(pd, st)], 256, 256, 8)
        plan.step(dict(ADAMW_HP, lr=lr), t)
        lr *= 0.5
        torch.cuda.synchronize()
        for a, b, s in zip(pw, pd, st):
            assert _same(a, b)
            assert _same(opt.state[a]["v_codes"], s["v_codes"])
            assert _same(opt.state[a]["m_codes"], s["m_codes"])


def test_adamw_state_dict_round_trip_and_closure(mods):
    import torch
    _, optim = mods
    shapes = [(128, 256), (512,)]
    pa, pb = _params(shapes, 20), _params(shapes, 20)
    oa = optim.AdamW(pa, v_bits=16, v_block=128)
    for t in (1, 2):
        _grads(pa, t, 900)
        oa.step()
    import io
    buf = io.BytesIO()
    torch.save(oa.state_dict(), buf)  # a checkpoint: state_dict() holds live references
    buf.seek(0)
    sd = torch.load(buf, weights_only=False)
    for p, q in zip(pa, pb):
        q.data.copy_(p.data)
    ob = optim.AdamW(pb, v_bits=16, v_block=128)
    ob.load_state_dict(sd)
    for p in pb:
        assert ob.state[p]["v_codes"].dtype == torch.int16
        assert ob.state[p]["m_codes"].dtype == torch.int8
    _grads(pa, 3, 900)
    _grads(pb, 3, 900)
    calls = []
    oa.step(lambda: calls.append(1) or torch.tensor(0.0))
    ob.step()
    torch.cuda.synchronize()
    assert calls == [1]
    for p, q in zip(pa, pb):
        assert _same(p, q)


def test_migrate_al8_to_al16_keeps_decoded_state(mods):
    """Sec. 6.2 per-role precision: re-coding a trained V from AL8 to AL16
    keeps every decoded value within AL16's half log-step of the AL8 value."""
    import torch
    B, optim = mods
    p = _params([(256, 512)], 30)
    opt = optim.AdamW(p)
    for t in (1, 2, 3):
        _grads(p, t, 700)
        opt.step()
    st = opt.state[p[0]]
    before = torch.empty(p[0].numel(), dtype=torch.float32, device="cuda")
    B.al_decode(st["v_codes"], st["v_meta"], 256, 8, before)
    opt.migrate_bits("v_bits", 16)
    assert opt.param_groups[0]["v_bits"] == 16 and st["v_codes"].dtype == torch.int16
    after = torch.empty_like(before)
    B.al_decode(st["v_codes"], st["v_meta"], 256, 16, after)
    b, a = before.cpu().numpy().astype(np.float64), after.cpu().numpy().astype(np.float64)
    assert np.array_equal(b == 0, a == 0)
    meta = st["v_meta"].cpu().numpy().reshape(-1, 2)
    step = np.repeat(meta[:, 1], 256)[: b.size] / 65534.0  # log2 step of AL16 per block
    nz = b > 0
    assert np.all(np.abs(np.log2(a[nz]) - np.log2(b[nz])) <= 0.5 * step[nz] * (1 + 1e-6) + 1e-7)
    _grads(p, 4, 700)
    opt.step()  # keeps stepping with AL16 states


def test_adafactor_and_came_wrappers_match_direct_calls(mods):
    import torch
    B, optim = mods
    shapes = [(256, 384), (384,)]
    for kind in ("adafactor", "came"):
        pw, pd = _params(shapes, 40), _params(shapes, 40)
        opt = optim.Adafactor(pw) if kind == "adafactor" else optim.CAME(pw)
        for t in (1, 2):
            _grads(pw, t, 300)
            _grads(pd, t, 300)
            opt.step()
            for i, p in enumerate(pd):
                rows, cols = (p.shape[0], p.shape[1]) if p.dim() == 2 else (1, p.numel())
                st = opt.state[pw[i]]
                if t == 1:
                    ref = {k: torch.zeros_like(v) for k, v in st.items() if torch.is_tensor(v)}
                    pd[i]._ref = ref
                ref = pd[i]._ref
                if kind == "adafactor":
                    ws = torch.empty(B.al_workspace_size(B.AL_OP_ADAFACTOR, rows, cols),
                                     dtype=torch.uint8, device="cuda")
                    hp = {k: opt.param_groups[0][k] for k in ("lr", "eps1", "clip_d", "decay_rate",
                                                              "beta1", "weight_decay", "log_floor")}
                    B.al_adafactor_step(p.data, p.grad, rows, cols, ref["r_codes"], ref["r_meta"],
                                        ref["c_codes"], ref["c_meta"], 16, 128, ref["m_codes"],
                                        ref["m_absmax"], 256, hp, t, ws)
                else:
                    ws = torch.empty(B.al_workspace_size(B.AL_OP_CAME, rows, cols),
                                     dtype=torch.uint8, device="cuda")
                    g = opt.param_groups[0]
                    hp = dict(lr=g["lr"], beta1=g["betas"][0], beta2=g["betas"][1],
                              beta3=g["betas"][2], eps1=g["eps"][0], eps2=g["eps"][1],
                              clip_d=g["clip_d"], weight_decay=g["weight_decay"],
                              log_floor_v=g["log_floor_v"], log_floor_c=g["log_floor_c"])
                    B.al_came_step(p.data, p.grad, rows, cols, ref["vr_codes"], ref["vr_meta"],
                                   ref["vc_codes"], ref["vc_meta"], 16, 128, ref["cr_codes"],
                                   ref["cr_meta"], ref["cc_codes"], ref["cc_meta"], 16, 128,
                                   ref["m_codes"], ref["m_absmax"], 256, hp, t, ws)
            torch.cuda.synchronize()
            for a, b in zip(pw, pd):
                assert _same(a, b), (kind, t)


def test_apollo_wrapper_grouped_step_and_routing(mods):
    """Matrices go through the grouped APOLLO step with the wrapper's own
    projections (checked against a direct plan fed the same projections);
    a vector parameter is routed to the quantized AdamW step."""
    import torch
    B, optim = mods
    shapes = [(256, 512), (512, 256), (256,)]
    pw, pd = _params(shapes, 60), _params(shapes, 60)
    opt = optim.Apollo(pw, lr=1e-4, rank=128, proj_gap=2)
    vec_before = pw[2].detach().clone()
    ref = None
    for t in (1, 2, 3):
        _grads(pw, t, 800)
        _grads(pd, t, 800)
        opt.step()
        if ref is None:
            ref = [{k: torch.zeros_like(v) for k, v in opt.state[p].items()
                    if torch.is_tensor(v) and k != "proj"} for p in pw[:2]]
        mats = [dict(p=pd[i].data, g=pd[i].grad, rows=pd[i].shape[0], cols=pd[i].shape[1],
                     proj=opt.state[pw[i]]["proj"], **ref[i]) for i in range(2)]
        hp = dict(lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, alpha=1.0, weight_decay=0.0,
                  norm_growth_gamma=0.0, log_floor=opt.param_groups[0]["log_floor"], rank=128)
        B.ApolloPlan(mats, 128, 8).step(hp, t)
        torch.cuda.synchronize()
        for i in range(2):
            assert _same(pw[i], pd[i]), (i, t)
    assert not _same(pw[2], vec_before)  # the vector was stepped (by AdamW)
    assert "proj" not in opt.state[pw[2]]
    sd = opt.state_dict()
    assert "adamw" in sd


def test_wrappers_reject_cpu_parameters(mods):
    import torch
    _, optim = mods
    p = torch.nn.Parameter(torch.zeros(16))
    p.grad = torch.zeros(16)
    with pytest.raises(ValueError):
        optim.AdamW([p]).step()


def test_g1_grouping_fp32_roles(mods):
    """Sec. 6.1's G1: 1-D tensors, biases, norms, embeddings and the LM head
    get unquantized states (v_bits 32: fp32 m and v; fac_bits 32: fp32
    factors), the rest the AL path; the FP32 AdamW group equals the oracle's
    unquantized step bit for bit."""
    import torch
    import oracle as ora
    B, optim = mods

    class Tiny(torch.nn.Module):
        def __init__(self):
            super().__init__()
            self.embed_tokens = torch.nn.Embedding(64, 32)
            self.proj = torch.nn.Linear(32, 48)
            self.norm = torch.nn.LayerNorm(48)
            self.lm_head = torch.nn.Linear(48, 64, bias=False)

    torch.manual_seed(0)
    model = Tiny().cuda()
    groups = optim.g1_param_groups(model.named_parameters(), dict(v_bits=32))
    names = {id(p): n for n, p in model.named_parameters()}
    assert [names[id(p)] for p in groups[0]["params"]] == ["proj.weight"]
    assert len(groups[1]["params"]) == 5 and groups[1]["v_bits"] == 32
    opt = optim.AdamW(groups, lr=1e-3, weight_decay=0.01)
    ref = {n: p.detach().cpu().numpy().ravel().copy() for n, p in model.named_parameters()}
    mv = {n: (np.zeros(r.size, np.float32), np.zeros(r.size, np.float32)) for n, r in ref.items()}
    for t in (1, 2, 3):
        for i, p in enumerate(model.parameters()):
            p.grad = torch.from_numpy(wl.gaussian_grad(tuple(p.shape), 1e-3, 50 * t + i)).cuda()
        for n, p in model.named_parameters():
            if n != "proj.weight":
                g = p.grad.cpu().numpy().ravel()
                ora.adamw_step(ref[n], g, mv[n][0], None, mv[n][1], None, 256, 256, 32,
                               dict(ADAMW_HP, lr=1e-3), t)
        opt.step()
        torch.cuda.synchronize()
        for n, p in model.named_parameters():
            if n != "proj.weight":
                assert np.array_equal(ref[n].view(np.uint32),
                                      p.detach().cpu().numpy().ravel().view(np.uint32)), (n, t)
    st = opt.state[model.norm.weight]
    assert st["m_codes"].dtype == torch.float32 and st["v_codes"].dtype == torch.float32
    assert opt.state[model.proj.weight]["v_codes"].dtype == torch.uint8
    # Adafactor G1: fp32 factors for the protected group
    opt2 = optim.Adafactor(optim.g1_param_groups(model.named_parameters(), dict(fac_bits=32)),
                           beta1=0.0)
    opt2.step()
    assert opt2.state[model.lm_head.weight]["r_codes"].dtype == torch.float32
    assert opt2.state[model.proj.weight]["r_codes"].dtype == torch.int16
    # CAME FP32-C: confidence factors fp32, second moment AL16
    opt3 = optim.CAME(model.parameters(), c_bits=32)
    opt3.step()
    st3 = opt3.state[model.proj.weight]
    assert st3["cr_codes"].dtype == torch.float32 and st3["vr_codes"].dtype == torch.int16
    assert torch.all(st3["cr_codes"] > 0)


@pytest.mark.parametrize("kind", ["AdamW", "CAME", "Apollo", "Adafactor"])
def test_wrappers_hold_no_gradients(mods, kind):
    """A training loop that frees its gradients every step
    (zero_grad(set_to_none=True), torch's default) gets fresh gradient
    tensors at new addresses: the cached plans are keyed on parameter and
    state addresses and rebind the gradients, so over 100 steps no plan is
    added and device memory stays flat after the second step."""
    import torch
    _, optim = mods
    shapes = [(256, 512), (128, 256), (512,)] if kind != "Apollo" else [(256, 512), (128, 256)]
    params = _params(shapes, 40)
    opt = {"AdamW": lambda: optim.AdamW(params),
           "CAME": lambda: optim.CAME(params),
           "Adafactor": lambda: optim.Adafactor(params),
           "Apollo": lambda: optim.Apollo(params, rank=128)}[kind]()
    gen = torch.Generator(device="cuda")
    gen.manual_seed(5)
    base = None
    for step in range(1, 101):
        opt.zero_grad(set_to_none=True)
        for p in params:
            p.grad = torch.randn(p.shape, device="cuda", generator=gen) * 1e-3
        opt.step()
        if step == 2:
            torch.cuda.synchronize()
            base = torch.cuda.memory_allocated()
            nplans = len(opt._plans)
    torch.cuda.synchronize()
    assert torch.cuda.memory_allocated() == base
    assert len(opt._plans) == nplans <= 1
    assert all(torch.isfinite(p).all() for p in params)


# -------------------------------------------------- wrappers vs the oracle --
def _np(t):
    import torch
    x = t.detach().cpu()
    if x.dtype == torch.int16:
        return x.numpy().view(np.uint16)
    return x.numpy()


def _set_grads(params, t, seed):
    import torch
    gs = []
    for i, p in enumerate(params):
        g = wl.student_t_grad(tuple(p.shape), 1e-3, 3.0, 0.05, seed + 100 * t + i)
        p.grad = torch.from_numpy(g).cuda()
        gs.append(g.ravel())
    return gs


def test_adamw_wrapper_with_g1_grouping_matches_oracle(mods):
    """optim.AdamW over G1 groups (Sec. 6.1: one-dimensional tensors, biases,
    norms and embeddings keep fp32 states, the rest AL8 V + UF8 M), 10 steps
    against the oracle's step per tensor: AL8/UF8 codes and block constants
    bit for bit, fp32-role states and parameters bit for bit, AL-path
    parameters within 1e-5 of |p| plus the step sizes."""
    import torch
    import oracle as ora
    from gpu_util import params_off, step_size
    _, optim = mods
    named = [("layer.weight", (64, 300)), ("layer.bias", (300,)), ("norm.weight", (512,)),
             ("embed.weight", (100, 64)), ("mlp.weight", (37, 111))]
    params = _params([s for _, s in named], 60)
    groups = optim.g1_param_groups(zip([n for n, _ in named], params), dict(v_bits=32))
    opt = optim.AdamW(groups, lr=1e-3, weight_decay=0.01)
    protected = {id(p) for g in groups if g.get("v_bits") == 32 for p in g["params"]}
    assert len(protected) == 3
    host = []
    for p in params:
        n = p.numel()
        raw = id(p) in protected
        host.append(dict(p=_np(p).ravel().copy(), raw=raw,
                         m=np.zeros(n, np.float32 if raw else np.int8),
                         ma=None if raw else np.zeros((n + 255) // 256, np.float32),
                         v=np.zeros(n, np.float32 if raw else np.uint8),
                         vm=None if raw else np.zeros(2 * ((n + 255) // 256), np.float32),
                         steps=np.zeros(n)))
    for t in range(1, 11):
        gs = _set_grads(params, t, 3000)
        opt.step()
        for h, g in zip(host, gs):
            before = h["p"].copy()
            ora.adamw_step(h["p"], g, h["m"], h["ma"], h["v"], h["vm"], 256, 256,
                           32 if h["raw"] else 8, ADAMW_HP, t)
            h["steps"] += step_size(h["p"], before, ADAMW_HP)
    torch.cuda.synchronize()
    for p, h in zip(params, host):
        st = opt.state[p]
        if h["raw"]:
            for want, got in ((h["p"], p), (h["m"], st["m_codes"]), (h["v"], st["v_codes"])):
                assert np.array_equal(want.view(np.uint8), _np(got).ravel().view(np.uint8))
        else:
            for want, key in ((h["m"], "m_codes"), (h["ma"], "m_absmax"), (h["v"], "v_codes"),
                              (h["vm"], "v_meta")):
                assert np.array_equal(want.view(np.uint8), _np(st[key]).view(np.uint8)), key
            assert params_off(h["p"], _np(p).ravel(), h["steps"]) == 0


@pytest.mark.parametrize("kind", ["Adafactor", "CAME"])
def test_factored_wrappers_match_oracle(mods, kind):
    """optim.Adafactor (AL16 factors, UF8 momentum) and optim.CAME (AL16 V
    and C, UF8 momentum) over two matrices and a vector (a 1 x n matrix),
    10 steps against the oracle's step per matrix: every code, block
    constant and parameter bit for bit."""
    import torch
    import oracle as ora
    _, optim = mods
    shapes = [(64, 300), (300,), (256, 128)]
    params = _params(shapes, 70)
    opt = optim.CAME(params) if kind == "CAME" else optim.Adafactor(params)
    g0 = opt.param_groups[0]
    host = []
    for p, s in zip(params, shapes):
        rows, cols = (s[0], s[1]) if len(s) == 2 else (1, s[0])
        n = rows * cols
        h = dict(p=_np(p).ravel().copy(), rows=rows, cols=cols,
                 mc=np.zeros(n, np.int8), ma=np.zeros((n + 255) // 256, np.float32))
        for k, ln in (("vr", rows), ("vc", cols), ("cr", rows), ("cc", cols)):
            h[k] = np.zeros(ln, np.uint16)
            h[k + "m"] = np.zeros(2 * ((ln + 127) // 128), np.float32)
        host.append(h)
    for t in range(1, 11):
        gs = _set_grads(params, t, 5000)
        opt.step()
        for h, g in zip(host, gs):
            if kind == "CAME":
                b1, b2, b3 = g0["betas"]
                hp = dict(lr=g0["lr"], beta1=b1, beta2=b2, beta3=b3, eps1=g0["eps"][0],
                          eps2=g0["eps"][1], clip_d=g0["clip_d"],
                          weight_decay=g0["weight_decay"], log_floor_v=g0["log_floor_v"],
                          log_floor_c=g0["log_floor_c"])
                ora.came_step(h["p"], g, h["rows"], h["cols"], h["vr"], h["vrm"], h["vc"],
                              h["vcm"], 16, 128, h["cr"], h["crm"], h["cc"], h["ccm"], 16, 128,
                              h["mc"], h["ma"], 256, hp, t)
            else:
                hp = {k: g0[k] for k in ("lr", "eps1", "clip_d", "decay_rate", "beta1",
                                          "weight_decay", "log_floor")}
                ora.adafactor_step(h["p"], g, h["rows"], h["cols"], h["vr"], h["vrm"], h["vc"],
                                   h["vcm"], 16, 128, h["mc"], h["ma"], 256, hp, t)
    torch.cuda.synchronize()
    keys = ({"vr": "vr_codes", "vrm": "vr_meta", "vc": "vc_codes", "vcm": "vc_meta",
             "cr": "cr_codes", "crm": "cr_meta", "cc": "cc_codes", "ccm": "cc_meta"}
            if kind == "CAME" else
            {"vr": "r_codes", "vrm": "r_meta", "vc": "c_codes", "vcm": "c_meta"})
    keys.update(mc="m_codes", ma="m_absmax")
    for p, h in zip(params, host):
        st = opt.state[p]
        assert np.array_equal(h["p"].view(np.uint32), _np(p).ravel().view(np.uint32))
        for hk, sk in keys.items():
            assert np.array_equal(h[hk].view(np.uint8), _np(st[sk]).view(np.uint8)), (kind, sk)


def test_apollo_wrapper_matches_oracle(mods):
    """optim.Apollo: a matrix stepped through the grouped APOLLO launch with
    the wrapper's own seeded projection, against the oracle's quantized
    APOLLO step with that projection over 10 steps (displacement within
    1e-4 of the oracle's: the projections accumulate differently, as in the
    direct tests), and a vector routed to the quantized AdamW step (codes
    and block constants bit for bit)."""
    import torch
    import oracle as ora
    from gpu_util import params_off, step_size
    _, optim = mods
    params = _params([(256, 512), (512,)], 80)
    opt = optim.Apollo(params, rank=128, lr=1e-4)
    mat, vec = params
    hp = dict(lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, alpha=1.0, weight_decay=0.0,
              norm_growth_gamma=0.0, log_floor=opt.param_groups[0]["log_floor"], rank=128)
    hm = dict(p=_np(mat).ravel().copy(), mc=np.zeros(512 * 128, np.int8),
              ma=np.zeros(512, np.float32), vc=np.zeros(512 * 128, np.uint8),
              vm=np.zeros(1024, np.float32))
    p0 = hm["p"].copy()
    hv = dict(p=_np(vec).ravel().copy(), mc=np.zeros(512, np.int8), ma=np.zeros(2, np.float32),
              vc=np.zeros(512, np.uint8), vm=np.zeros(4, np.float32), steps=np.zeros(512))
    ahp = dict(ADAMW_HP, lr=1e-4, weight_decay=0.0)
    for t in range(1, 11):
        gs = _set_grads(params, t, 7000)
        opt.step()
        P = _np(opt.state[mat]["proj"]).copy()
        ora.apollo_step(hm["p"], gs[0], 256, 512, P, hm["mc"], hm["ma"], 128, hm["vc"],
                        hm["vm"], 8, 128, 0.0, hp, t)
        before = hv["p"].copy()
        ora.adamw_step(hv["p"], gs[1], hv["mc"], hv["ma"], hv["vc"], hv["vm"], 256, 256, 8,
                       ahp, t)
        hv["steps"] += step_size(hv["p"], before, ahp)
    torch.cuda.synchronize()
    pm = _np(mat).ravel().astype(np.float64)
    disp = np.linalg.norm(pm - p0) and (np.linalg.norm((pm - p0) - (hm["p"] - p0))
                                        / np.linalg.norm(hm["p"] - p0))
    assert disp < 1e-4, disp
    st = opt._adamw.state[vec]
    for want, key in ((hv["mc"], "m_codes"), (hv["ma"], "m_absmax"), (hv["vc"], "v_codes"),
                      (hv["vm"], "v_meta")):
        assert np.array_equal(want.view(np.uint8), _np(st[key]).view(np.uint8)), key
    assert params_off(hv["p"], _np(vec).ravel(), hv["steps"]) == 0
