"""The exact fp16 tcgen05 product path against the oracle and against the integer-MMA path.

Codes are centered (c - 128) into fp16, exact; products and sums of up to 1024 of them are exact in
the fp32 tensor-memory accumulator; longer K is accumulated in chunks drained into int32. Every
result must equal the oracle's bit for bit (int32 accumulator and recovered fp32)."""
import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qnn():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1607_04683_gb300 import build, qnn as q
    build.build()
    q.lib()
    torch.cuda.set_device(0)
    return q


def gpu(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _run(qnn, ca, pa, ga, ra, cw, pw, cs, nb=1, bias=None):
    return qnn.qnn_qmatmul(gpu(ca), qnn.params_tensor(pa), ga, gpu(ra), gpu(cw), qnn.params_tensor(pw), gpu(cs),
                           n_blocks=nb, bias=None if bias is None else gpu(bias), want_acc=True)


TC_SHAPES = [(1, 8, 1), (3, 300, 40), (128, 256, 64), (130, 260, 100), (257, 2000, 500), (384, 512, 1024),
             (200, 136, 1025), (129, 257, 2048), (256, 256, 8192)]


@pytest.mark.parametrize("M,N,K", TC_SHAPES)
def test_tc_path_bit_exact(qnn, M, N, K, monkeypatch):
    g = np.random.Generator(np.random.PCG64(M * 31 + N * 7 + K))
    A = g.normal(0.1, 1.0, (M, K)).astype(np.float32)
    nb = 4 if N % 4 == 0 else 1
    Ws = [g.uniform(-s, s, (N // nb, K)).astype(np.float32) for s in np.linspace(0.05, 0.4, nb)]
    ca, pa, ra = oracle.quantize(A, oracle.PER_ROW)
    parts = [oracle.quantize(w, oracle.PER_MATRIX) for w in Ws]
    cw = np.concatenate([p[0] for p in parts])
    pw = np.concatenate([p[1] for p in parts])
    cs = np.concatenate([p[2] for p in parts])
    bias = g.normal(0, 1, N).astype(np.float32)
    ref = oracle.qmatmul(ca, pa, 1, cw, pw, n_blocks=nb, bias=bias)
    # tile widths 64 and 128 take the row epilogue (two blocks per SM) when K <= 1024, 256 the
    # staged one; K > 1024 always drains chunks through the staged epilogue
    for path, bn in (("tc", None), ("tc", "64"), ("tc", "128"), ("tc", "256"), ("imma", None)):
        monkeypatch.setenv("QNN_QGEMM", path)
        if bn:
            monkeypatch.setenv("QNN_TC_BN", bn)
        else:
            monkeypatch.delenv("QNN_TC_BN", raising=False)
        Y, acc = _run(qnn, ca, pa, 1, ra, cw, pw, cs, nb, bias)
        assert qnn.device_status() == qnn.QNN_OK
        assert np.array_equal(acc.cpu().numpy(), ref["acc"]), (path, bn)
        assert np.array_equal(Y.cpu().numpy(), ref["y"]), (path, bn)


@pytest.mark.parametrize("K", [1024, 1025, 2048])
@pytest.mark.parametrize("a_code,w_code", [(0, 0), (255, 255), (0, 255)])
def test_tc_extreme_codes_at_the_exactness_limit(qnn, K, a_code, w_code, monkeypatch):
    # centered values +-128 / 127 everywhere: |sum| reaches 2^24 at K = 1024, the fp32 limit
    monkeypatch.setenv("QNN_QGEMM", "tc")
    M, N = 128, 256
    ca = np.full((M, K), a_code, np.uint8)
    cw = np.full((N, K), w_code, np.uint8)
    p = np.zeros(1, qnn.QPARAMS_DTYPE)
    p[0] = (0.0, 1.0, 255.0, 0)
    ra = ca.astype(np.int64).sum(1).astype(np.int32)
    cs = cw.astype(np.int64).sum(1).astype(np.int32)
    Y, acc = _run(qnn, ca, p, 0, ra, cw, p, cs)
    assert np.all(acc.cpu().numpy() == a_code * w_code * K)


def _adversarial_rows(g, n, K):
    """Centered code rows (s = c - 128) that drive partial sums of s_a s_w towards +-2^24 and then
    add small odd terms: runs of -128 or 127 (products +-16384, +-16256, 16129) followed by +-1 and
    +-3, sign patterns alternating in blocks of 16 (one MMA's K step) and of 64 (one k-block),
    random extremes, and random extremes that end in small odd values."""
    rows = []
    for i in range(n):
        kind = i % 6
        s = np.empty(K, np.int64)
        if kind == 0:    # a long run of -128, then a tail of +-1 / +-3
            s[:] = -128
            tail = min(K, 16 + (i % 48))
            s[K - tail:] = g.choice([-3, -1, 1, 3], tail)
        elif kind == 1:  # a run of 127 (products of 16129 or -16256 against -128), odd tail
            s[:] = 127
            tail = min(K, 1 + (i % 31))
            s[K - tail:] = g.choice([-1, 1], tail)
        elif kind == 2:  # sign alternating in blocks of 16
            s[:] = np.where((np.arange(K) // 16) % 2 == 0, -128, 127)
            s[-1] = 1
        elif kind == 3:  # sign alternating in blocks of 64, an odd term in each block
            s[:] = np.where((np.arange(K) // 64) % 2 == 0, 127, -128)
            s[63::64] = 3
        elif kind == 4:  # random extremes
            s[:] = g.choice([-128, 127], K)
        else:            # random extremes, then random small odd values
            s[:] = g.choice([-128, 127], K)
            tail = min(K, 8 + (i % 100))
            s[K - tail:] = g.choice([-3, -1, 1, 3], tail)
        rows.append(s + 128)
    return np.array(rows, np.uint8)


@pytest.mark.parametrize("K", [256, 512, 1000, 1024, 1025, 2048])
def test_tc_adversarial_partial_sums_bit_exact(qnn, K, monkeypatch):
    # the fp16 datapath is exact only if the tensor-memory accumulator keeps every integer up to
    # 2^24: large partial sums followed by small odd terms, with mixed signs, must come out exact
    # at K-chunk lengths 256, 512, 1024 and across chunk boundaries
    monkeypatch.delenv("QNN_TC_BN", raising=False)
    g = np.random.Generator(np.random.PCG64(K + 17))
    M, N = 192, 144
    ca = _adversarial_rows(g, M, K)
    cw = _adversarial_rows(g, N, K)
    cw = np.concatenate([cw[:N // 2], 255 - cw[N // 2:]])  # sign-flipped half: sums towards -2^24 too
    p = np.zeros(1, qnn.QPARAMS_DTYPE)
    p[0] = (0.0, 1.0, 255.0, 0)
    ra = ca.astype(np.int64).sum(1).astype(np.int32)
    cs = cw.astype(np.int64).sum(1).astype(np.int32)
    ref = oracle.qmatmul(ca, p, 0, cw, p)
    cent = (ca.astype(np.int64) - 128) @ (cw.astype(np.int64) - 128).T
    # the centered sums come close to the largest a chunk of min(K, 1024) terms can reach (2^24)
    assert np.abs(cent).max() > 0.9 * min(K, 1024) * (1 << 14)
    assert np.count_nonzero(cent % 2) > 0           # and end odd
    for path in ("tc", "imma"):
        monkeypatch.setenv("QNN_QGEMM", path)
        Y, acc = _run(qnn, ca, p, 0, ra, cw, p, cs)
        assert qnn.device_status() == qnn.QNN_OK
        assert np.array_equal(acc.cpu().numpy(), ref["acc"]), path
        assert np.array_equal(Y.cpu().numpy(), ref["y"]), path


@pytest.mark.parametrize("K", [64, 1000, 3000])
def test_tc_large_offsets_bit_exact(qnn, K, monkeypatch):
    """Rows with a narrow range far from zero have large offsets z (eq. 2), so the offset-applied
    sums S of eq. (1) reach far beyond 2^22 and the recovery converts them the wide way."""
    monkeypatch.delenv("QNN_TC_BN", raising=False)
    g = np.random.Generator(np.random.PCG64(K))
    M, N = 300, 200
    A = (1000.0 + g.uniform(0.0, 0.5, (M, K))).astype(np.float32)
    A[::7] = g.normal(0, 1, (A[::7].shape)).astype(np.float32)  # and some ordinary rows
    W = g.uniform(-0.1, 0.1, (N, K)).astype(np.float32)
    ca, pa, ra = oracle.quantize(A, oracle.PER_ROW)
    cw, pw, cs = oracle.quantize(W, oracle.PER_MATRIX)
    assert np.abs(pa["z"]).max() > 1 << 18
    ref = oracle.qmatmul(ca, pa, 1, cw, pw)
    for path in ("tc", "imma"):
        monkeypatch.setenv("QNN_QGEMM", path)
        Y, acc = _run(qnn, ca, pa, 1, ra, cw, pw, cs)
        assert qnn.device_status() == qnn.QNN_OK
        assert np.array_equal(acc.cpu().numpy(), ref["acc"]), path
        assert np.array_equal(Y.cpu().numpy(), ref["y"]), path
        # without the raw accumulator the full 16-column blocks take the fast recovery: 32-bit sums
        # for the ordinary rows, 64-bit ones for the large-offset rows
        Y2, _ = qnn.qnn_qmatmul(gpu(ca), qnn.params_tensor(pa), 1, gpu(ra), gpu(cw), qnn.params_tensor(pw), gpu(cs))
        assert np.array_equal(Y2.cpu().numpy(), ref["y"]), path


def test_s64_to_f32_rounds_to_nearest_even(qnn):
    """The recovery's int64 -> fp32 conversion against the host's IEEE conversion: every magnitude,
    exact halfway cases (ties to even) and their neighbours, and the carry into a new leading bit."""
    g = np.random.Generator(np.random.PCG64(11))
    parts = [g.integers(-(1 << 62), 1 << 62, 200000, dtype=np.int64)]
    for top in range(20, 63):  # random values with a given leading-bit position
        parts.append(g.integers(1 << top, 1 << (top + 1), 2000, dtype=np.int64))
    ties = []
    for sh in range(1, 40):
        m = g.integers(1 << 23, 1 << 24, 200, dtype=np.int64)
        base = (m << sh) + (1 << (sh - 1))  # exactly halfway between two fp32 values
        ties += [base, base - 1, base + 1]
    parts += ties
    parts.append(np.array([(1 << 24) - 1, 1 << 24, (1 << 24) + 1, (1 << 31) - 1, 1 << 31, -(1 << 31), -(1 << 31) - 1,
                           (1 << 63) - 1, -(1 << 63), ((1 << 24) - 1) << 39, (((1 << 24) - 1) << 39) + (1 << 38)],
                          dtype=np.int64))
    v = np.concatenate(parts)
    v = np.concatenate([v, -v[v != -(1 << 63)]])
    got = qnn.selftest_s64_to_f32(torch.from_numpy(v).cuda()).cpu().numpy()
    want = v.astype(np.float32)
    assert np.array_equal(got.view(np.int32), want.view(np.int32))


def test_paired_gate_functions_equal_the_scalar_ones(qnn):
    """The fused gate kernel computes E, sigma, tanh, the cell update and the recovery's quotient two
    cells at a time with paired fp32 instructions; every component must equal the one-value form bit
    for bit (else layer outputs would drift from the oracle). Inputs span the exponential's clamp
    range and beyond, with values at and next to the half-integer multiples of ln 2 where the
    reduction's rounding decides n."""
    g = np.random.Generator(np.random.PCG64(21))
    parts = [g.uniform(-100, 100, 1 << 21), g.uniform(-10, 10, 1 << 21), g.uniform(-1, 1, 1 << 20),
             g.normal(0, 1e-3, 1 << 18)]
    ln2 = np.log(2.0)
    half = (np.arange(-130, 130) + 0.5) * ln2
    near = np.concatenate([np.nextafter(half.astype(np.float32), np.float32(s)) for s in (-np.inf, np.inf)] +
                          [half.astype(np.float32)])
    v = np.concatenate([p.astype(np.float32) for p in parts] + [near, np.float32([0.0, -0.0, 87.0, -87.0, 88.0, -88.0])])
    if v.size % 2:
        v = np.concatenate([v, np.float32([1.0])])
    assert qnn.selftest_pair_functions(torch.from_numpy(v).cuda()) == 0
    # the pairs the other way round too
    w = v.reshape(-1, 2)[:, ::-1].copy().ravel()
    assert qnn.selftest_pair_functions(torch.from_numpy(w).cuda()) == 0
