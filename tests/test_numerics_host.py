"""CPU parity of the CUDA library's codec arithmetic (host build) with the
oracle.

The library evaluates Eq. (3)-(5) with fp32/two-float fast paths and an FP64
fallback near rounding boundaries (alq_numerics.h). Built for the host, the
same source must reproduce the oracle's codes, bounds and decoded values bit
for bit, with rare fallbacks. The GPU build differs only in the hardware
log2 approximation used by the encoder's fast path (covered by the GPU
tests).
"""
import ctypes as C
import math
import os
import subprocess

import numpy as np
import pytest

import oracle as ora
from paper_2608_22322_gb300 import workloads as wl

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(ROOT, "paper_2608_22322_gb300", "csrc")
SRC = os.path.join(HERE, "numerics_host.cpp")
OUT = os.path.join(ROOT, "_build", "numerics_host.so")


@pytest.fixture(scope="module")
def lib():
    os.makedirs(os.path.dirname(OUT), exist_ok=True)
    deps = [SRC, os.path.join(CSRC, "alq_numerics.h"), os.path.join(CSRC, "al_tables.inc")]
    if not os.path.exists(OUT) or any(os.path.getmtime(d) > os.path.getmtime(OUT) for d in deps):
        tmp = OUT + f".{os.getpid()}"
        subprocess.run(["g++", "-O2", "-std=c++17", "-ffp-contract=off", "-fno-fast-math",
                        "-shared", "-fPIC", "-I", CSRC, "-o", tmp, SRC], check=True)
        os.replace(tmp, OUT)
    L = C.CDLL(OUT)
    f32p = np.ctypeslib.ndpointer(np.float32, flags="C_CONTIGUOUS")
    L.alqn_log2_rn.restype = C.c_float
    L.alqn_log2_rn.argtypes = [C.c_float]
    L.alqn_log2_rn_fast.restype = C.c_float
    L.alqn_log2_rn_fast.argtypes = [C.c_float, C.POINTER(C.c_int)]
    L.alqn_block_params.argtypes = [C.c_float, C.c_float, C.c_float,
                                    C.POINTER(C.c_float), C.POINTER(C.c_float)]
    L.alqn_level.argtypes = [C.c_float, C.c_float, C.c_int, C.c_float,
                             C.POINTER(C.c_float), C.POINTER(C.c_float)]
    L.alqn_al8_decode.argtypes = [np.ctypeslib.ndpointer(np.uint8), C.c_int64, C.c_float,
                                  C.c_float, f32p, C.POINTER(C.c_int64)]
    L.alqn_al_quantize.argtypes = [f32p, C.c_int64, C.c_float, C.c_float, C.c_int,
                                   np.ctypeslib.ndpointer(np.uint32), C.POINTER(C.c_int64)]
    L.alqn_al_quantize_ff.argtypes = L.alqn_al_quantize.argtypes
    return L


def test_log2_rn_matches_double_rounding(lib):
    r = wl.rng(1)
    xs = np.concatenate([
        np.exp2(r.uniform(-126, 127, 200000)).astype(np.float32),
        (1 + r.uniform(-1e-3, 1e-3, 20000)).astype(np.float32),  # near 1
        np.float32(2.0) ** np.arange(-126, 127, dtype=np.float32),  # exact powers
        np.array([1e-42, 3e-39, 1.0], np.float32),  # subnormal, tiny, exact 1
    ])
    for x in xs:
        assert lib.alqn_log2_rn(float(x)) == np.float32(math.log2(float(x))), x


def test_log2_rn_fast_certifies_only_correct_roundings(lib):
    """The hardware-log2 fast path of the block bounds: whenever it certifies
    its result, the result is (float)log2((double)x); it certifies most
    values of the second-moment range (|log2 x| in [16, 64)) and declines
    near 1, for subnormals and for ties it cannot separate."""
    r = wl.rng(2)
    xs = np.concatenate([
        np.exp2(r.uniform(-126, 127, 200000)).astype(np.float32),
        np.exp2(r.uniform(-64, -16, 100000)).astype(np.float32),
        (1 + r.uniform(-1e-3, 1e-3, 20000)).astype(np.float32),
        np.float32(2.0) ** np.arange(-126, 127, dtype=np.float32),
        np.array([1e-42, 3e-39, 1.0], np.float32),
    ])
    ok = C.c_int(0)
    certified = in_range = cert_in_range = 0
    for x in xs:
        got = lib.alqn_log2_rn_fast(float(x), C.byref(ok))
        want = np.float32(math.log2(float(x)))
        if ok.value:
            certified += 1
            assert got == want, x
        if 16.0 <= abs(float(want)) < 64.0:
            in_range += 1
            cert_in_range += ok.value
        if x < np.float32(2.0) ** -126 or abs(float(x) - 1.0) < 1e-3:
            assert not ok.value, x
    assert cert_in_range > 0.8 * in_range, (cert_in_range, in_range)


def test_block_params_match_oracle(lib):
    r = wl.rng(2)
    floor_ = np.float32(math.log2(1e-16))
    for _ in range(20000):
        x = np.exp2(r.uniform(-70, 20, 8)).astype(np.float32)
        if r.random() < 0.1:
            x[:] = x[0]  # degenerate: all equal
        lm, de, _ = ora.al_block_meta(x, float(floor_))
        a, b = C.c_float(), C.c_float()
        lib.alqn_block_params(float(x.min()), float(x.max()), float(floor_), C.byref(a), C.byref(b))
        assert (np.float32(a.value), np.float32(b.value)) == (lm, de)


def test_level_two_float_accuracy(lib):
    """Table levels: |hi + lo - 2^(l_min + k Delta / 254)| < 2^-44 relative
    (reference in Python decimal arithmetic)."""
    from decimal import Decimal, getcontext
    getcontext().prec = 50
    ln2 = Decimal(2).ln()
    r = wl.rng(3)
    worst = 0.0
    for _ in range(3000):
        lmin = np.float32(r.uniform(-96, 40))
        delta = np.float32(r.uniform(1e-3, min(222.0, 126.0 - float(lmin))))
        k = int(r.integers(-1, 255))
        hi, lo = C.c_float(), C.c_float()
        lib.alqn_level(float(lmin), float(delta), k, 254.0, C.byref(hi), C.byref(lo))
        y = Decimal(float(lmin)) + Decimal(k) * Decimal(float(delta)) / 254
        ref = (y * ln2).exp()
        got = Decimal(hi.value) + Decimal(lo.value)
        worst = max(worst, float(abs(got - ref) / ref))
    assert worst < 2.0 ** -44, worst


def test_al8_decode_tables_match_oracle(lib):
    r = wl.rng(4)
    codes = np.arange(256, dtype=np.uint8)
    fb_total = C.c_int64(0)
    n_total = 0
    for _ in range(4000):
        lmin = np.float32(r.uniform(-96, 30))
        delta = np.float32(r.choice([r.uniform(0.01, 2), r.uniform(2, 60),
                                     r.uniform(60, 120)]))
        if lmin + delta > 126:
            continue
        out = np.zeros(256, np.float32)
        lib.alqn_al8_decode(codes, 256, float(lmin), float(delta), out, C.byref(fb_total))
        want = np.array([ora.al_dequantize(int(q), lmin, delta, 8) for q in codes], np.float32)
        np.testing.assert_array_equal(out.view(np.uint32), want.view(np.uint32))
        n_total += 256
    assert fb_total.value < n_total * 1e-4, (fb_total.value, n_total)


@pytest.mark.parametrize("bits", [8, 16])
def test_al_quantize_fast_matches_oracle(lib, bits):
    r = wl.rng(5 + bits)
    fb = C.c_int64(0)
    n_total = 0
    floor_ = np.float32(math.log2(1e-16))
    for _ in range(400):
        spread = float(r.choice([0.5, 5.0, 20.0, 60.0]))
        x = np.exp2(r.uniform(-40, -40 + spread, 512)).astype(np.float32)
        x[r.random(512) < 0.05] = 0.0
        lm, de, _ = ora.al_block_meta(x, float(floor_))
        q = np.zeros(512, np.uint32)
        lib.alqn_al_quantize(x, 512, float(lm), float(de), bits, q, C.byref(fb))
        want = np.array([ora.al_quantize(float(v), lm, de, bits) for v in x], np.uint32)
        np.testing.assert_array_equal(q, want)
        n_total += 512
    limit = 2e-3 if bits == 8 else 0.2  # AL16's 65534 levels exceed fp32 resolution
    assert fb.value < n_total * limit, (fb.value, n_total)


@pytest.mark.parametrize("bits", [8, 16])
def test_al_quantize_two_float_matches_oracle(lib, bits):
    """The two-float Eq. (4) that refines the values the fp32 fast path
    cannot decide, on values placed within 1e-4 of the half-integers of t
    (where the fast path gives up) and on random ones, equals the oracle's
    double expression; it leaves a tiny fraction to FP64."""
    r = wl.rng(40 + bits)
    Lm2 = (1 << bits) - 2
    floor_ = np.float32(math.log2(1e-16))
    und = C.c_int64(0)
    n_total = 0
    for _ in range(300):
        spread = float(r.choice([0.5, 5.0, 20.0, 60.0]))
        lo = float(r.uniform(-60, -20))
        x = np.exp2(r.uniform(lo, lo + spread, 512)).astype(np.float32)
        lm, de, _ = ora.al_block_meta(x, float(floor_))
        # half of them next to a code boundary: t = k + 0.5 +- 1e-4
        k = r.integers(0, Lm2, 256) + 0.5 + r.uniform(-1e-4, 1e-4, 256)
        x[:256] = np.exp2(float(lm) + k * float(de) / Lm2).astype(np.float32)
        q = np.zeros(512, np.uint32)
        lib.alqn_al_quantize_ff(x, 512, float(lm), float(de), bits, q, C.byref(und))
        want = np.array([ora.al_quantize(float(v), lm, de, bits) for v in x], np.uint32)
        np.testing.assert_array_equal(q, want)
        n_total += 512
    assert und.value < n_total * 1e-3, (und.value, n_total)
