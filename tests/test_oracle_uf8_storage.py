"""Pins of the oracle's UF8 momentum code and of the AL storage formula.

UF8 (Sec. 4.3, Sec. 5.6): the paper fixes a uniform signed 8-bit code with no
sign flips; these tests check the half-step error bound, sign preservation,
the endpoint codes and the all-zero block, and compare codes against exact
rational rounding computed independently in Python integers.

Storage (Sec. 4.4, Eq. (7)): the numbers printed in Sec. 4.4, Sec. 5.3,
Sec. 5.5 and the TinyLlama-1.1B results table of Sec. 6.2 are reproduced from
tests/golden/paper_storage.json.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle as ora
from paper_2608_22322_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_storage.json")


def _momentum(n, seed, scale=1e-4, zero_frac=0.05):
    r = wl.rng(seed)
    m = (r.standard_normal(n) * scale).astype(np.float32)
    m[r.random(n) < zero_frac] = 0.0
    return m


@pytest.mark.parametrize("block", [32, 256, 2048])
def test_uf8_error_bound_and_signs(block):
    m = _momentum(7 * block + 3, block)
    m[block:2 * block] = 0.0
    codes, absmax = ora.uf8_encode(m, block)
    mh = ora.uf8_decode(codes, absmax, block)
    for b in range(absmax.size):
        sl = slice(b * block, (b + 1) * block)
        s = float(absmax[b])
        assert s == float(np.max(np.abs(m[sl])))
        # half a code step, plus fp32 rounding of the product and of s/127
        assert np.max(np.abs(mh[sl] - m[sl])) <= s / 254 * (1 + 1e-6) + 2 * s * 2.0 ** -24
    assert np.all(np.sign(codes) * np.sign(m) >= 0)   # no sign flips
    assert np.all(np.abs(codes.astype(int)) <= 127)
    assert not codes[block:2 * block].any() and absmax[1] == 0
    np.testing.assert_array_equal(mh[m == 0], 0)


def test_uf8_absmax_element_is_127():
    m = _momentum(256, 3)
    k = int(np.argmax(np.abs(m)))
    codes, _ = ora.uf8_encode(m, 256)
    assert abs(int(codes[k])) == 127 and np.sign(codes[k]) == np.sign(m[k])


def test_uf8_matches_exact_rational_rounding():
    """q = round(127 m / s) computed in exact rationals, except where the fp32
    evaluation of m*(127/s) sits within 1e-4 of a half-integer."""
    m = _momentum(64 * 256, 8)
    codes, absmax = ora.uf8_encode(m, 256)
    skipped = 0
    for i in range(m.size):
        s = Fraction(float(absmax[i // 256]))
        if s == 0:
            assert codes[i] == 0
            continue
        exact = Fraction(127) * Fraction(float(m[i])) / s
        fl = math.floor(exact)
        frac = exact - fl
        if abs(frac - Fraction(1, 2)) < Fraction(1, 10000):
            skipped += 1
            continue
        want = fl + (1 if frac > Fraction(1, 2) else 0)
        assert int(codes[i]) == want
    assert skipped < m.size * 1e-3


def test_uf8_tiny_block_scaling():
    """Blocks with absmax below 2^-120 (scaled by 2^64 internally) code the
    same as the exact rational rounding."""
    m = (_momentum(256, 12, scale=1.0) * np.float32(2.0 ** -126)).astype(np.float32)
    codes, absmax = ora.uf8_encode(m, 256)
    s = Fraction(float(absmax[0]))
    for v, q in zip(m, codes):
        exact = Fraction(127) * Fraction(float(v)) / s
        if abs(exact - math.floor(exact) - Fraction(1, 2)) < Fraction(1, 1000):
            continue
        assert int(q) == round(exact)


# ------------------------------------------------------------ storage -----
def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


def test_golden_bits_per_element():
    g = _golden()
    for row in g["al8_bits_per_element"]:
        n = 1 << 30
        bits = 8 * ora.al_state_bytes(n, row["block"], 8) / n
        assert round(bits, row["decimals"]) == row["value"], row


def test_golden_metadata_bytes_per_element():
    g = _golden()
    for row in g["metadata_bytes_per_element"]:
        n = 1 << 30
        meta = (ora.al_state_bytes(n, row["block"], 8) - n) / n
        if row.get("scales_per_block") == 1:  # bnb-style single fp32 scale
            meta /= 2
        assert round(meta, row["decimals"]) == row["value"], row


def test_golden_v_state_mib():
    g = _golden()
    for row in g["al8_state_mib_1p1e9"]:
        mib = ora.al_state_bytes(int(1.1e9), row["block"], 8) / 2 ** 20
        assert round(mib, 1) == row["value"], row


def test_golden_tinyllama_state_mib():
    """Optimizer-state MiB of the results table (Sec. 6.2) from the 201
    TinyLlama-1.1B tensor shapes: FP32 AdamW (two fp32 states), AL8 (B=2048)
    + UF8 (B=256) with the 45 one-dimensional norm vectors kept in fp32, and
    the FP32 factored Adafactor reference."""
    g = _golden()["tinyllama_state_mib"]
    tensors = wl.tinyllama_tensors()
    n_all = sum(wl.numel(s) for _, s in tensors)
    assert n_all == g["params"]
    fp32_adamw = 8 * n_all / 2 ** 20
    assert round(fp32_adamw, 1) == g["adamw_fp32"]
    q = 0
    for _, s in tensors:
        n = wl.numel(s)
        if len(s) == 1:
            q += 8 * n  # fp32 m and v
        else:
            q += ora.al_state_bytes(n, 2048, 8) + n + 4 * ((n + 255) // 256)
    assert round(q / 2 ** 20, 1) == g["adamw_al8_uf8_b2048"]
    fac = sum((s[0] + s[1]) if len(s) == 2 else s[0] for _, s in tensors)
    assert round(4 * fac / 2 ** 20, 1) == g["adafactor_fp32_factored"]
