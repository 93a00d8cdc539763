"""GPU parity of the AL and UF8 codec kernels with the oracle (bit-exact).

Sec. 4.1 Eq. (3)-(5), Sec. 4.3. The same seeded fp32 inputs go to the CUDA
library (through the C ABI) and to the oracle; codes, block metadata and
decoded values must agree bit for bit, over every supported block size, both
bit widths, ragged lengths, all-zero / constant / below-floor blocks and
-0.0 entries.
"""
import numpy as np
import pytest

import oracle as ora
from gpu_util import FLOOR, bytes_equal, gpu_available, state_mix
from paper_2608_22322_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not gpu_available(), reason="needs a CUDA GPU")]


@pytest.fixture(scope="module")
def B():
    from paper_2608_22322_gb300 import binding
    return binding


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


@pytest.mark.parametrize("bits", [8, 16])
@pytest.mark.parametrize("block", [128, 256, 512, 1024, 2048, 4096])
def test_al_encode_bit_exact(B, bits, block):
    import torch
    n = 5 * 4096 + 3 * block + 13
    x = state_mix(n, block, seed=block + bits)
    codes, meta = ora.al_encode(x, block, bits, FLOOR)
    tc = torch.zeros(n, dtype=torch.uint8 if bits == 8 else torch.int16, device="cuda")
    tm = torch.zeros(2 * B.al_num_blocks(n, block), dtype=torch.float32, device="cuda")
    B.al_encode(_dev(x), block, bits, FLOOR, tc, tm)
    torch.cuda.synchronize()
    assert bytes_equal(meta, tm.cpu().numpy()) == 0
    got = tc.cpu().numpy().view(ora.code_dtype(bits))
    assert int(np.sum(got != codes)) == 0


def _subnormal_mix(n, block, seed):
    """Blocks whose minimum positive value is subnormal (the encoder's
    exact path for a whole segment), mixed with zeros, -0.0 and normal
    values reaching up to 2^20, next to blocks of normal values only."""
    r = wl.rng(seed)
    x = np.exp2(r.uniform(-40, 20, n)).astype(np.float32)
    nb = (n + block - 1) // block
    for b in range(0, nb, 3):
        lo, hi = b * block, min(n, (b + 1) * block)
        k = hi - lo
        sub = (r.integers(1, 1 << 23, k, dtype=np.uint32)).view(np.float32)
        pick = r.random(k)
        seg = x[lo:hi].copy()
        seg[pick < 0.3] = sub[pick < 0.3]
        seg[(pick >= 0.3) & (pick < 0.4)] = 0.0
        seg[(pick >= 0.4) & (pick < 0.45)] = -0.0
        if b % 2 == 0:
            seg[:] = np.where(pick < 0.5, sub, seg)  # mostly tiny values
        x[lo:hi] = seg
    return x


@pytest.mark.parametrize("bits", [8, 16])
@pytest.mark.parametrize("block", [128, 256, 2048])
@pytest.mark.parametrize("floor", [FLOOR, -160.0])
def test_al_encode_subnormal_blocks(B, bits, block, floor):
    """Subnormal minima put l_min below -126 with a low floor: zeros must
    still code as 0 and every value must match Eq. (4) in double."""
    import torch
    n = 12 * block + 37
    x = _subnormal_mix(n, block, seed=block + bits)
    codes, meta = ora.al_encode(x, block, bits, floor)
    tc = torch.zeros(n, dtype=torch.uint8 if bits == 8 else torch.int16, device="cuda")
    tm = torch.zeros(2 * B.al_num_blocks(n, block), dtype=torch.float32, device="cuda")
    B.al_encode(_dev(x), block, bits, floor, tc, tm)
    torch.cuda.synchronize()
    assert bytes_equal(meta, tm.cpu().numpy()) == 0
    got = tc.cpu().numpy().view(ora.code_dtype(bits))
    assert int(np.sum(got != codes)) == 0
    assert np.all(got[x == 0] == 0)
    assert float(meta[0::2].min()) < -126.0 or floor > -126.0


@pytest.mark.parametrize("bits", [8, 16])
@pytest.mark.parametrize("block", [128, 256, 2048])
def test_al_decode_bit_exact(B, bits, block):
    import torch
    n = 40 * 4096 + 77
    x = state_mix(n, block, seed=7 + block)
    codes, meta = ora.al_encode(x, block, bits, FLOOR)
    want = ora.al_decode(codes, meta, block, bits)
    out = torch.empty(n, dtype=torch.float32, device="cuda")
    B.al_decode(_dev(codes.view(np.uint8 if bits == 8 else np.int16)), _dev(meta), block,
                bits, out)
    torch.cuda.synchronize()
    assert bytes_equal(want, out.cpu().numpy()) == 0


def test_al8_decode_all_codes_many_blocks(B):
    """Every AL8 code under 20000 random (l_min, Delta): exercises the
    two-float table path and its FP64 fallback at fp32 rounding boundaries."""
    import torch
    r = wl.rng(11)
    nb = 20000
    lmin = r.uniform(-96, 20, nb).astype(np.float32)
    delta = np.minimum(r.choice([0.3, 5, 20, 60, 120], nb) * r.uniform(0.5, 1.5, nb),
                       126 - lmin).astype(np.float32)
    meta = np.stack([lmin, delta], 1).ravel().astype(np.float32)
    codes = np.tile(np.arange(256, dtype=np.uint8), nb)
    want = ora.al_decode(codes, meta, 256, 8)
    out = torch.empty(codes.size, dtype=torch.float32, device="cuda")
    B.al_decode(_dev(codes), _dev(meta), 256, 8, out)
    torch.cuda.synchronize()
    assert bytes_equal(want, out.cpu().numpy()) == 0


@pytest.mark.parametrize("block", [128, 256, 4096])
def test_uf8_bit_exact(B, block):
    import torch
    n = 9 * 4096 + 5
    r = wl.rng(block)
    m = (r.standard_normal(n) * 1e-4).astype(np.float32)
    m[r.random(n) < 0.05] = 0.0
    m[block:2 * block] = 0.0                                  # all-zero block
    m[3 * block:4 * block] *= np.float32(2.0 ** -110)         # tiny block (2^64 scaling)
    codes, absmax = ora.uf8_encode(m, block)
    tc = torch.zeros(n, dtype=torch.int8, device="cuda")
    ta = torch.zeros(B.al_num_blocks(n, block), dtype=torch.float32, device="cuda")
    B.uf8_encode(_dev(m), block, tc, ta)
    out = torch.empty(n, dtype=torch.float32, device="cuda")
    B.uf8_decode(_dev(codes), _dev(absmax), block, out)
    torch.cuda.synchronize()
    assert bytes_equal(codes, tc.cpu().numpy()) == 0
    assert bytes_equal(absmax, ta.cpu().numpy()) == 0
    assert bytes_equal(ora.uf8_decode(codes, absmax, block), out.cpu().numpy()) == 0


def test_encode_fast_path_every_mantissa(B):
    """The encoder's fp32 fast path bounds its error assuming the hardware
    log2 approximation is within 2^-21 of log2(m) on m in [1, 2). Blocks whose
    values span [1, 2) (l_min = 0, Delta ~ 1, so t = 254 log2 m) run every fp32
    mantissa through it; all codes must equal the oracle's."""
    import torch
    block = 4096
    m = (np.arange(1 << 23, dtype=np.uint32) | np.uint32(0x3F800000)).view(np.float32)
    parts = [np.concatenate([np.float32([1.0, 1.9999999]), m[lo:lo + block - 2]])
             for lo in range(0, m.size, block - 2)]
    x = np.concatenate(parts).astype(np.float32)
    codes, meta = ora.al_encode(x, block, 8, -200.0)
    tc = torch.zeros(x.size, dtype=torch.uint8, device="cuda")
    tm = torch.zeros(2 * B.al_num_blocks(x.size, block), dtype=torch.float32, device="cuda")
    B.al_encode(_dev(x), block, 8, -200.0, tc, tm)
    torch.cuda.synchronize()
    assert bytes_equal(meta, tm.cpu().numpy()) == 0
    assert int(np.sum(tc.cpu().numpy() != codes)) == 0


def test_codec_empty_and_tiny_inputs(B):
    """n = 0 is a no-op; n = 1..7 (one partial block, shorter than a
    vector) round-trips exactly as the oracle codes it."""
    import torch
    z = torch.zeros(0, device="cuda")
    B.al_encode(z, 256, 8, FLOOR, torch.zeros(0, dtype=torch.uint8, device="cuda"), z)
    B.al_decode(torch.zeros(0, dtype=torch.uint8, device="cuda"), z, 256, 8, z)
    for n in range(1, 8):
        x = state_mix(n, 256, seed=900 + n)
        x[0] = 3.5e-7
        codes, meta = ora.al_encode(x, 256, 8, FLOOR)
        tc = torch.zeros(n, dtype=torch.uint8, device="cuda")
        tm = torch.zeros(2, dtype=torch.float32, device="cuda")
        B.al_encode(_dev(x), 256, 8, FLOOR, tc, tm)
        out = torch.empty(n, dtype=torch.float32, device="cuda")
        B.al_decode(tc, tm, 256, 8, out)
        torch.cuda.synchronize()
        assert bytes_equal(meta, tm.cpu().numpy()) == 0, n
        assert np.array_equal(tc.cpu().numpy(), codes), n
        assert bytes_equal(ora.al_decode(codes, meta, 256, 8), out.cpu().numpy()) == 0, n
