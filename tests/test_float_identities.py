"""Float identities the kernels rely on to compute the same values as the oracle's operations.

The gate nonlinearities (sigma = 1/(E(-x) + 1), tanh = 1 - 2/(E(2x) + 1), Sec. 3.1 cell with the
pinned exponential) are evaluated on the GPU from the correctly rounded reciprocal r = RN(1/d):
sigma is r itself, tanh is 1 - 2 r. The oracle divides. These checks, in IEEE float32 on the host
(numpy rounds every operation to nearest even, subnormals included), pin that the two agree bit
for bit over every d the gates can meet: d = E + 1 with E in [E(-87), E(88)].
"""
import numpy as np

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
