"""The integer fp32 <-> fp64 conversions of the fp64 gradient accumulation.

The kernels widen every fp32 run sum to fp64 before the fp64 reduction and
round the fp64 accumulator back to fp32 for the optimizer, both in integer
arithmetic (no FP64-pipe conversion).  These tests call the same device
routines through pss_check_convert and compare them bit for bit with the
IEEE-754 conversions numpy performs (exact widening; round to nearest, ties to
even), over every class of input: normals, subnormals, signed zeros,
infinities, NaNs, halfway cases, and the edges of the fp32 range.
"""
import ctypes

import numpy as np
import pytest

from paper_2207_10731_gb300 import binding
from tests import gpu_util as gu

pytestmark = pytest.mark.gpu


def _run(direction, host_in, out_dtype):
    t = gu.torch()
    lib = binding.load_library()
    d_in = t.from_numpy(host_in).cuda()
    d_out = t.empty(host_in.shape[0], dtype=out_dtype, device="cuda")
    rc = lib.pss_check_convert(direction, gu.ctypes_ptr(d_in), gu.ctypes_ptr(d_out),
                               host_in.shape[0], ctypes.c_void_p(int(t.cuda.current_stream().cuda_stream)))
    assert rc == binding.PSS_OK
    t.cuda.synchronize()
    return d_out.cpu().numpy()


def _same_bits_or_both_nan(got, want, utype):
    nan = np.isnan(want)
    assert np.array_equal(np.isnan(got), nan)
    np.testing.assert_array_equal(got[~nan].view(utype), want[~nan].view(utype))


def test_widen_is_exact_for_every_class():
    rng = np.random.default_rng(7)
    bits = rng.integers(0, 1 << 32, size=1 << 20, dtype=np.uint64).astype(np.uint32)
    special = np.array([0x00000000, 0x80000000, 0x00000001, 0x80000001, 0x007fffff, 0x00400000,
                        0x00800000, 0x7f7fffff, 0xff7fffff, 0x7f800000, 0xff800000, 0x7fc00000,
                        0x7f800001, 0x3f800000, 0xbf800000], dtype=np.uint32)
    sub = rng.integers(1, 1 << 23, size=4096, dtype=np.uint64).astype(np.uint32)
    x = np.concatenate([bits, special, sub, sub | np.uint32(0x80000000)]).view(np.float32)
    got = _run(0, x, gu.torch().float64)
    _same_bits_or_both_nan(got, x.astype(np.float64), np.uint64)


def test_narrow_rounds_to_nearest_even_for_every_class():
    rng = np.random.default_rng(11)
    raw = rng.integers(0, 1 << 63, size=1 << 20, dtype=np.uint64)
    raw[: 1 << 19] |= np.uint64(1) << np.uint64(63)
    # values inside and just around the fp32 range (exponents 1023 +- 160)
    e = rng.integers(1023 - 160, 1023 + 130, size=1 << 20, dtype=np.uint64)
    m = rng.integers(0, 1 << 52, size=1 << 20, dtype=np.uint64)
    near = (e << np.uint64(52)) | m
    # exact halfway cases: the 29 dropped bits are 1000...0 (ties), with odd and
    # even kept fractions, in the normal and the subnormal range of fp32
    keep = rng.integers(0, 1 << 23, size=4096, dtype=np.uint64)
    ev = rng.integers(1023 - 126, 1023 + 127, size=4096, dtype=np.uint64)
    ties = (ev << np.uint64(52)) | (keep << np.uint64(29)) | (np.uint64(1) << np.uint64(28))
    sub_e = rng.integers(1023 - 150, 1023 - 126, size=4096, dtype=np.uint64)
    sub = (sub_e << np.uint64(52)) | (keep << np.uint64(29))
    special = np.array([0.0, -0.0, np.inf, -np.inf, np.nan, 5e-324, -5e-324, 1e-300,
                        float(np.finfo(np.float32).max), 3.4028235677973366e38,
                        3.4028235677973362e38, 1.401298464324817e-45, 7.006492321624085e-46,
                        7.006492321624087e-46, 2.1019476964872256e-45, 1.1754942106924411e-38,
                        1.1754943508222875e-38, 1.0, -1.0, 1.0000000596046448,
                        1.0000001788139343], dtype=np.float64)
    x = np.concatenate([raw.view(np.float64), near.view(np.float64), ties.view(np.float64),
                        sub.view(np.float64), special])
    got = _run(1, x, gu.torch().float32)
    with np.errstate(over="ignore", invalid="ignore"):
        want = x.astype(np.float32)
    _same_bits_or_both_nan(got, want, np.uint32)
