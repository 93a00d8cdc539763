"""Controlled fidelity probes on the GPU (Sec. 5): the relative update error
of Eq. (2) and the temporal drift of an AL-coded second-moment EMA, on
synthetic log-normal regimes.

These are diagnostics, not the optimizer path: the quantized quantities come
from the library (the AL codec and the fused AdamW step), while the fp32
reference trajectories and the update operator U(V, G) = G / (sqrt(V) + eps)
(Adam's use of the second moment) are plain torch arithmetic on the device.
The paper does not state its generators, so only orderings and the paper's
qualitative claims are comparable (adaptive AL8 below 1% single-step update
error in every regime, Sec. 5.2; smaller blocks drift less, Sec. 5.6).

    python -m paper_2608_22322_gb300.probes        # prints the probe tables
"""
from __future__ import annotations

import math

import torch

from . import binding as B

# log2-space regimes of the second moment: (mean, spread within a block,
# spread of the block offsets) of log2 V. Sec. 5.2 names narrow, medium and
# wide regimes by their relative sampled log-spans without printing their
# parameters; its adaptive AL8 errors (0.039%, 0.688%, 0.704%) correspond to
# per-block spans of about 1, 17 and 18 octaves, so "wide" is read as wide
# across blocks (where one fixed floor fails) with a medium span inside each
# block. These parameters are this library's choices.
REGIMES = {"narrow": (-24.0, 0.15, 0.0), "medium": (-24.0, 2.5, 0.0), "wide": (-24.0, 2.5, 8.0)}


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def lognormal_state(n: int, regime: str, seed: int, block: int = 2048,
                    device="cuda") -> torch.Tensor:
    """V with log2 V = mu + s_b Z_block + s_w Z_element for the regime's
    (mu, s_w, s_b) (fp32, all positive)."""
    mu, s_w, s_b = REGIMES[regime]
    gen = _gen(seed, device)
    z = torch.empty(n, dtype=torch.float32, device=device).normal_(0.0, 1.0, generator=gen)
    nb = (n + block - 1) // block
    zb = torch.empty(nb, dtype=torch.float32, device=device).normal_(0.0, 1.0, generator=gen)
    return torch.exp2(mu + s_w * z + s_b * zb.repeat_interleave(block)[:n])


def update_error(u_hat: torch.Tensor, u: torch.Tensor, eps: float = 1e-30) -> float:
    """Eq. (2): ||U(S_hat, G) - U(S, G)||_2 / (||U(S, G)||_2 + eps), in double."""
    d = (u_hat.double() - u.double()).norm().item()
    return d / (u.double().norm().item() + eps)


def single_step_update_error(regime: str, block: int = 2048, bits: int = 8,
                             n: int = 1 << 22, seed: int = 0, eps: float = 1e-8,
                             device="cuda") -> float:
    """Relative update error of U = G / (sqrt(V) + eps) when V is replaced by
    its AL round trip (Eq. (3)-(5)), G ~ N(0, sqrt(V)) elementwise."""
    v = lognormal_state(n, regime, seed, block, device)
    g = torch.empty_like(v).normal_(0.0, 1.0, generator=_gen(seed + 1, device)) * v.sqrt()
    codes = torch.empty(n, dtype=torch.uint8 if bits == 8 else torch.int16, device=device)
    meta = torch.empty(2 * ((n + block - 1) // block), dtype=torch.float32, device=device)
    floor = -126.0
    B.al_encode(v, block, bits, floor, codes, meta)
    v_hat = torch.empty_like(v)
    B.al_decode(codes, meta, block, bits, v_hat)
    return update_error(g / (v_hat.sqrt() + eps), g / (v.sqrt() + eps))


def ema_drift(steps: int = 5000, block: int = 2048, bits: int = 8, n: int = 1 << 20,
              regime: str = "medium", beta1: float = 0.9, beta2: float = 0.999,
              eps: float = 1e-8, seed: int = 0, device="cuda", grad_fn=None,
              return_state: bool = False):
    """A `steps`-long Adam-style EMA of fresh gradients whose per-block scale
    follows the regime (Sec. 5.6): the quantized second moment comes from the
    fused AdamW step (lr = 0, AL-coded V, UF8 M), the reference from float64
    EMAs of the same gradients. Returns (V drift, steady-state update error) in the sense of
    Eq. (2): ||V_hat - V|| / ||V|| and the relative error of
    M / (sqrt(V) + eps) with fp32 M against the same with V_hat.
    grad_fn(t), if given, supplies step t's gradient (a device tensor of n
    fp32 values) instead of the regime's draws; return_state adds the final
    (m_codes, m_absmax, v_codes, v_meta)."""
    nb = (n + block - 1) // block
    scale = (None if grad_fn is not None else
             lognormal_state(nb, regime, seed, 1, device).sqrt().repeat_interleave(block)[:n])
    p = torch.zeros(n, dtype=torch.float32, device=device)
    mc = torch.zeros(n, dtype=torch.int8, device=device)
    ma = torch.zeros((n + 255) // 256, dtype=torch.float32, device=device)
    vc = torch.zeros(n, dtype=torch.uint8 if bits == 8 else torch.int16, device=device)
    vm = torch.zeros(2 * nb, dtype=torch.float32, device=device)
    v = torch.zeros(n, dtype=torch.float64, device=device)
    m = torch.zeros(n, dtype=torch.float64, device=device)
    g = torch.empty(n, dtype=torch.float32, device=device)
    hp = dict(lr=0.0, beta1=beta1, beta2=beta2, eps=eps, weight_decay=0.0,
              log_floor=float(torch.tensor(math.log2(eps * eps), dtype=torch.float32)))
    gen = _gen(seed + 7, device)
    for t in range(1, steps + 1):
        if grad_fn is not None:
            g = grad_fn(t)
        else:
            g.normal_(0.0, 1.0, generator=gen).mul_(scale)
        B.al_adamw_step(p, g, mc, ma, vc, vm, 256, block, bits, hp, t)
        gd = g.double()
        v.mul_(beta2).add_(gd * gd, alpha=1.0 - beta2)
        m.mul_(beta1).add_(gd, alpha=1.0 - beta1)
    v_hat = torch.empty(n, dtype=torch.float32, device=device)
    B.al_decode(vc, vm, block, bits, v_hat)
    v_hat = v_hat.double()
    drift = update_error(v_hat, v)
    upd = update_error(m / (v_hat.sqrt() + eps), m / (v.sqrt() + eps))
    if return_state:
        return drift, upd, (mc, ma, vc, vm)
    return drift, upd


def main():
    print("single-step update error (Eq. (2), %), block 2048")
    print(f"{'regime':8s} {'AL8':>8s} {'AL16':>10s}")
    for r in REGIMES:
        e8 = single_step_update_error(r, 2048, 8)
        e16 = single_step_update_error(r, 2048, 16)
        print(f"{r:8s} {100 * e8:8.3f} {100 * e16:10.5f}")
    print("5K-step EMA (beta2 = 0.999), medium regime: V drift %, update error %")
    for blk in (256, 512, 1024, 2048):
        d, u = ema_drift(5000, blk, 8)
        print(f"block {blk:5d}  AL8  drift {100 * d:7.3f}  update {100 * u:7.3f}")


if __name__ == "__main__":
    main()
