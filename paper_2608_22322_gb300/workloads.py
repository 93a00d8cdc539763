"""Seeded synthetic inputs shaped like the paper's workloads.

This module holds shapes and random draws only -- none of the method's
arithmetic -- so the oracle-side tests and the CUDA-side tests and benchmark
can share it. Host arrays come from numpy's PCG64; the large benchmark inputs
are drawn on the device with torch's seeded CUDA generator.

Workloads (the paper trains TinyLlama-1.1B, Sec. 6.1; the optimizer step only
sees parameter- and gradient-shaped arrays, so synthetic draws of those
shapes stand in for the WikiText-103 gradients):
  adamw_single   one 256x1024 fp32 tensor; grads N(0, 1e-3) with 10% exact
                 zeros (persistent mask) and 2% of the rows all-zero (dormant).
  adafactor      one 4096x4096 weight; grads N(0, 1e-3) times a per-column
                 lognormal(0, 1) scale, 5% exact zeros.
  came           22 matrices 2048x5632; grads 1e-3 * Student-t(nu = 3), 5%
                 exact zeros.
  tinyllama      the 201 tensors of TinyLlama-1.1B (22 layers, hidden 2048,
                 MLP 5632, 32 query / 4 KV heads of dim 64, vocab 32000,
                 untied embeddings, RMSNorm vectors): 1,100,048,384 params;
                 params N(0, 0.02) (norm vectors 1.0), grads N(0, 1e-3) with
                 1% exact zeros.
  apollo         the 154 attention/MLP matrices of that model with a rank-256
                 Gaussian projection N(0, 1/r) rounded to bf16 per matrix.
"""
from __future__ import annotations

import numpy as np

SEED_BASE = 20260

# ------------------------------------------------------------- TinyLlama ----
TL_LAYERS = 22
TL_HIDDEN = 2048
TL_MLP = 5632
TL_VOCAB = 32000
TL_KV = 4 * 64  # 4 key/value heads of dim 64


def tinyllama_tensors():
    """[(name, shape)] of the 201 TinyLlama-1.1B parameter tensors."""
    out = [("embed_tokens", (TL_VOCAB, TL_HIDDEN))]
    for layer in range(TL_LAYERS):
        pre = f"layers.{layer}."
        out += [
            (pre + "q_proj", (TL_HIDDEN, TL_HIDDEN)),
            (pre + "k_proj", (TL_KV, TL_HIDDEN)),
            (pre + "v_proj", (TL_KV, TL_HIDDEN)),
            (pre + "o_proj", (TL_HIDDEN, TL_HIDDEN)),
            (pre + "gate_proj", (TL_MLP, TL_HIDDEN)),
            (pre + "up_proj", (TL_MLP, TL_HIDDEN)),
            (pre + "down_proj", (TL_HIDDEN, TL_MLP)),
            (pre + "input_layernorm", (TL_HIDDEN,)),
            (pre + "post_attention_layernorm", (TL_HIDDEN,)),
        ]
    out += [("norm", (TL_HIDDEN,)), ("lm_head", (TL_VOCAB, TL_HIDDEN))]
    return out


def tinyllama_matrices():
    """[(name, shape)] of the 154 attention/MLP matrices (APOLLO's set)."""
    keep = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj",
            "down_proj")
    return [(n, s) for n, s in tinyllama_tensors()
            if len(s) == 2 and n.split(".")[-1] in keep]


def numel(shape) -> int:
    return int(np.prod(shape))


# ---------------------------------------------------------------- configs ----
CONFIGS = {
    "adamw_single": dict(index=1, shape=(256, 1024), grad_std=1e-3,
                         zero_frac=0.10, dormant_row_frac=0.02,
                         lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8,
                         weight_decay=0.01, m_block=256, v_block=256, v_bits=8,
                         steps=10),
    "adafactor": dict(index=2, shape=(4096, 4096), grad_std=1e-3,
                      zero_frac=0.05, lr=1e-3, eps1=1e-30, clip_d=1.0,
                      decay_rate=-0.8, beta1=0.9, weight_decay=0.0,
                      fac_bits=16, fac_block=128, m_block=256, steps=20),
    "came": dict(index=3, n_mats=22, shape=(2048, 5632), grad_scale=1e-3,
                 nu=3.0, zero_frac=0.05, lr=1e-4, beta1=0.9, beta2=0.999,
                 beta3=0.9999, eps1=1e-30, eps2=1e-16, clip_d=1.0,
                 weight_decay=0.0, v_bits=16, v_block=128, c_bits=16,
                 c_block=128, m_block=256, steps=10),
    "tinyllama_adamw": dict(index=4, grad_std=1e-3, zero_frac=0.01,
                            lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8,
                            weight_decay=0.01, m_block=256, v_block=256,
                            v_bits=8, steps=10),
    "tinyllama_apollo": dict(index=5, grad_std=1e-3, rank=256, lr=1e-4,
                             beta1=0.9, beta2=0.999, eps=1e-8, alpha=1.0,
                             weight_decay=0.0, m_block=256, v_block=256,
                             v_bits=8, refresh=200, steps=10),
}


def rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


# ------------------------------------------------------------ host draws ----
def param_init(shape, seed: int, norm_vector_value: float = 1.0) -> np.ndarray:
    """N(0, 0.02) for matrices, a constant for 1-D norm vectors."""
    if len(shape) == 1:
        return np.full(shape, norm_vector_value, dtype=np.float32)
    return (rng(seed).standard_normal(shape) * 0.02).astype(np.float32)


def zero_mask(shape, frac: float, seed: int) -> np.ndarray:
    """Boolean mask of exact zeros (True = forced zero)."""
    return rng(seed).random(shape) < frac


def dormant_rows(n_rows: int, frac: float, seed: int) -> np.ndarray:
    """Indices of rows whose gradient is always zero."""
    k = max(1, int(round(n_rows * frac)))
    return np.sort(rng(seed).choice(n_rows, size=k, replace=False))


def gaussian_grad(shape, std: float, seed: int, mask=None) -> np.ndarray:
    g = (rng(seed).standard_normal(shape) * std).astype(np.float32)
    if mask is not None:
        g[mask] = 0.0
    return g


def lognormal_col_grad(shape, std: float, zero_frac: float, seed: int):
    r = rng(seed)
    g = r.standard_normal(shape) * std
    g *= np.exp(r.standard_normal((1, shape[1])))
    g[r.random(shape) < zero_frac] = 0.0
    return g.astype(np.float32)


def student_t_grad(shape, scale: float, nu: float, zero_frac: float, seed: int):
    r = rng(seed)
    g = r.standard_t(nu, size=shape) * scale
    g[r.random(shape) < zero_frac] = 0.0
    return g.astype(np.float32)


def gaussian_projection(rank: int, short: int, seed: int) -> np.ndarray:
    """fp32 N(0, 1/rank) draws of a [rank x short] projection."""
    return (rng(seed).standard_normal((rank, short)) / np.sqrt(rank)).astype(np.float32)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest even) and return the 16-bit patterns."""
    u = np.ascontiguousarray(x, np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


class AdamWSingle:
    """Host draws of the single-tensor AdamW workload (persistent mask)."""

    def __init__(self, shape=(256, 1024), seed=SEED_BASE + 1, zero_frac=0.10,
                 dormant_frac=0.02, grad_std=1e-3, redraw_mask=False):
        self.shape, self.seed = shape, seed
        self.zero_frac, self.grad_std = zero_frac, grad_std
        self.redraw_mask = redraw_mask
        self.p0 = param_init(shape, seed)
        self.mask = zero_mask(shape, zero_frac, seed + 7)
        self.dormant = dormant_rows(shape[0], dormant_frac, seed + 11)
        self.mask[self.dormant, :] = True

    def grad(self, t: int) -> np.ndarray:
        mask = self.mask
        if self.redraw_mask:
            mask = zero_mask(self.shape, self.zero_frac, self.seed + 1000 + t)
            mask[self.dormant, :] = True
        return gaussian_grad(self.shape, self.grad_std, self.seed + 100 + t, mask)


# ---------------------------------------------------------- device draws ----
def torch_device_normal_(t, std: float, seed: int):
    """Fill a CUDA tensor with N(0, std) from a seeded device generator."""
    import torch
    gen = torch.Generator(device=t.device)
    gen.manual_seed(seed)
    t.normal_(0.0, std, generator=gen)
    return t


def torch_device_zero_(t, frac: float, seed: int):
    """Zero a seeded random fraction of a CUDA tensor in place."""
    import torch
    gen = torch.Generator(device=t.device)
    gen.manual_seed(seed)
    drop = torch.rand(t.shape, device=t.device, generator=gen) < frac
    t.masked_fill_(drop, 0.0)
    return t
