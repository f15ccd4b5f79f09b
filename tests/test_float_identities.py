"""Float identities the kernels rely on to compute the same values as the oracle's operations.

The recovery of eq. (3) divides an exact integer sum S (|S| < 2^31) by Qa Qw. The tensor-core gate
kernel takes that quotient from the divisor's correctly rounded reciprocal r, computed once per
(row, gate): q = RN(S r), then RN(q + (S - q d) r) with the remainder formed exactly by a fused
multiply-add (the final step of Markstein's division). A C helper checks, with gcc's fmaf, that
this equals the IEEE quotient for every 24-bit numerator significand against 64 divisor
significands (all-ones and power-of-two neighbours among them) and on random integer/divisor pairs.
The softmax divides each E(l - max) in [2^-100, 1] by the row's sum in [1, C] the same way; random
pairs over those ranges (divisors up to 2^24) are checked too.

The gate nonlinearities (sigma = 1/(E(-x) + 1), tanh = 1 - 2/(E(2x) + 1), Sec. 3.1 cell with the
pinned exponential) are evaluated on the GPU from the correctly rounded reciprocal r = RN(1/d):
sigma is r itself, tanh is 1 - 2 r. The oracle divides. These checks, in IEEE float32 on the host
(numpy rounds every operation to nearest even, subnormals included), pin that the two agree bit
for bit over every d the gates can meet: d = E + 1 with E in [E(-87), E(88)].
"""
import os
import shutil
import subprocess
import tempfile

import numpy as np
import pytest

F = np.float32
D_MAX = F(1.0) + F(np.exp(np.float64(88.0)))  # above E(88) + 1 for any faithful E


def _ds(seed=3, n=200000):
    r = np.random.Generator(np.random.PCG64(seed))
    # log-uniform over [1, D_MAX], plus the ends, powers of two and their neighbours
    d = np.exp(r.uniform(0.0, np.log(np.float64(D_MAX)), n)).astype(F)
    p2 = np.ldexp(F(1.0), np.arange(0, 128)).astype(F)
    edges = np.concatenate([p2, np.nextafter(p2, F(np.inf)), np.nextafter(p2, F(0)),
                            np.array([1.0, D_MAX, np.nextafter(D_MAX, F(0))], F)])
    d = np.concatenate([d, edges]).astype(F)
    return d[(d >= F(1.0)) & (d <= D_MAX)]


def test_reciprocal_is_the_quotient_of_one():
    d = _ds()
    with np.errstate(under="ignore"):
        assert np.array_equal((F(1.0) / d).view(np.uint32), np.reciprocal(d).view(np.uint32))


def test_twice_the_reciprocal_is_the_quotient_of_two_while_normal():
    d = _ds()
    with np.errstate(under="ignore"):
        r = F(1.0) / d
        normal = r >= np.finfo(F).tiny
        assert np.count_nonzero(~normal) > 0  # the subnormal range is exercised too
        assert np.array_equal((F(2.0) * r)[normal].view(np.uint32), (F(2.0) / d)[normal].view(np.uint32))
        # where r is subnormal the quotient is tiny and tanh's 1 - q is 1 either way
        one_minus_a = F(1.0) - F(2.0) * r
        one_minus_b = F(1.0) - F(2.0) / d
        assert np.array_equal(one_minus_a.view(np.uint32), one_minus_b.view(np.uint32))
        assert np.all(one_minus_a[~normal] == F(1.0))


def test_identity_would_catch_a_wrong_scale():
    # a plausible slip (r rounded after scaling by a non-power of two) breaks the identity
    d = _ds(n=20000)
    with np.errstate(under="ignore"):
        assert not np.array_equal((F(3.0) * (F(1.0) / d)).view(np.uint32), (F(3.0) / d).view(np.uint32))


def test_quotient_from_the_reciprocal_is_the_ieee_quotient():
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = os.path.join(os.path.dirname(os.path.abspath(__file__)), "div_identity.c")
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "div_identity")
        subprocess.check_call([cc, "-O2", "-ffp-contract=off", "-fno-fast-math", "-o", exe, src, "-lm"])
        n, bad = (int(v) for v in subprocess.check_output([exe, "64", "20000000", "20000000"], text=True).split())
    assert n == 64 * (1 << 23) + 20000000 + 20000000
    assert bad == 0
