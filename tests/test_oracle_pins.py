"""Pins for the CPU oracle: each test checks the oracle against something other than itself —
closed forms derived by hand from the paper's definitions, the paper's stated invariants,
algebraic identities between different formulations, brute force, libm in double precision, and
a float64 textbook LSTM. A plausible mistake in the oracle (a dropped offset term, floor instead
of round, the Sec. 3 recovery instead of eq. (3), a swapped gate, a wrong sign) fails one of them.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_1607_04683_gb300 import inputs

F32 = np.float32


def f32(x):
    return float(np.float32(x))


# ------------------------------------------------------------------------------------------
# Quantizer: Sec. 3 "Quantizing", eq. (2), eq. (3)
# ------------------------------------------------------------------------------------------

def test_worked_example_symmetric_range():
    # V = {-1, 0, 0.5, 1}: R = 2, Q = 255/2 = 127.5 (exact in fp32); round(Q*vmin) = round(-127.5)
    # = -128 (half to even); eq. (2): round(Q v) + 128 = {0, 128, 192, 256}; the top code is
    # clamped to 255. Eq. (3): (c - 128)/127.5 = {-256/255, 0, 128/255, 254/255}.
    codes, p, sums = oracle.quantize(np.array([[-1.0, 0.0, 0.5, 1.0]], F32))
    assert p[0]["Q"] == 127.5 and p[0]["z"] == -128
    assert codes.tolist() == [[0, 128, 192, 255]]
    assert sums.tolist() == [575]
    rec = oracle.recover(codes[0], p[0])
    assert rec.tolist() == [f32(-256 / 255), 0.0, f32(128 / 255), f32(254 / 255)]


def test_worked_example_asymmetric_range():
    # V = {-0.5, 0.25, 1.75}: R = 2.25, Q = fl(255/2.25) = fl(113.333...) ; round(Q*(-0.5)) =
    # round(-56.67) = -57; codes round(Q v) + 57 = {0, 28 + 57, 198 + 57} = {0, 85, 255}.
    codes, p, _ = oracle.quantize(np.array([[-0.5, 0.25, 1.75]], F32))
    assert p[0]["Q"] == f32(255 / 2.25)
    assert p[0]["z"] == -57
    assert codes.tolist() == [[0, 85, 255]]


def test_min_to_zero_max_to_top_every_code_in_range():
    # Sec. 3: the range [Vmin, Vmax] is squeezed into [0, S], S = 255.
    rng = np.random.Generator(np.random.PCG64(11))
    for trial in range(3000):
        n = int(rng.integers(2, 64))
        kind = trial % 4
        if kind == 0:
            v = rng.uniform(-0.1, 0.1, n)
        elif kind == 1:
            a = rng.uniform(1e-3, 10.0)
            v = rng.uniform(-a, a, n)
            v[0], v[1] = -a, a  # exactly symmetric range: needs the nudge (reading R1)
        elif kind == 2:
            v = rng.normal(rng.uniform(-5, 5), rng.uniform(1e-2, 3), n)
        else:
            v = 1.0 / (1.0 + np.exp(-rng.normal(0, 2, n)))
        v = v.astype(F32)[None, :]
        codes, p, sums = oracle.quantize(v)
        assert codes[0, np.argmin(v)] == 0
        assert codes[0, np.argmax(v)] == 255
        assert codes.min() >= 0 and codes.max() <= 255
        assert sums[0] == int(codes.astype(np.int64).sum())


def test_recovery_error_at_most_half_step():
    # Eq. (2) then eq. (3): |v - v_hat| <= 0.5/Q, plus fp32 rounding of Q*v and of the recovery
    # divide (each at most 2^-24 relative) and the <= few-ulp change of Q from the nudge.
    rng = np.random.Generator(np.random.PCG64(12))
    for trial in range(400):
        n = 257
        lo = rng.uniform(-20, 20)
        hi = lo + rng.uniform(1e-2, 20)
        v = rng.uniform(lo, hi, n).astype(F32)
        codes, p, _ = oracle.quantize(v[None, :])
        Q, z = float(p[0]["Q"]), int(p[0]["z"])
        A = max(abs(Q * float(v.min())), abs(Q * float(v.max()))) + 256.0
        bound = (0.5 + A * 2.0 ** -20) / Q
        rec = (codes[0].astype(np.float64) + z) / Q
        assert np.max(np.abs(rec - v.astype(np.float64))) <= bound
        # the oracle's own fp32 recovery is within one more fp32 rounding
        rec32 = oracle.recover(codes[0, :16], p[0]).astype(np.float64)
        assert np.max(np.abs(rec32 - v[:16])) <= bound + np.abs(rec32).max() * 2.0 ** -23


def test_offset_consistency_removes_bias():
    # Sec. 3.1: quantizing with round(Q V) - round(Q Vmin) and recovering with eq. (3) is
    # consistent, so the mean error of many values spread uniformly over the range is ~0 (no bias).
    # The inconsistent recovery V' / Q + Vmin of Sec. 3 shifts every value by (z - Q Vmin)/Q.
    rng = np.random.Generator(np.random.PCG64(13))
    v = rng.uniform(-0.37, 0.81, 200000).astype(F32)
    codes, p, _ = oracle.quantize(v[None, :])
    Q, z = float(p[0]["Q"]), int(p[0]["z"])
    rec = (codes[0].astype(np.float64) + z) / Q
    err = rec - v
    assert abs(err.mean()) < 0.02 / Q
    naive = codes[0].astype(np.float64) / Q + float(p[0]["vmin"])
    shift = (z - Q * float(p[0]["vmin"])) / Q
    assert np.allclose((naive - v).mean() - err.mean(), -shift, atol=1e-9)


def test_power_of_two_scaling_leaves_codes_unchanged():
    rng = np.random.Generator(np.random.PCG64(14))
    for _ in range(200):
        v = rng.normal(rng.uniform(-2, 2), rng.uniform(0.1, 2), 100).astype(F32)
        c0, p0, _ = oracle.quantize(v[None, :])
        for k in (-7, -1, 1, 5):
            ck, pk, _ = oracle.quantize((v * F32(2.0 ** k))[None, :])
            assert np.array_equal(c0, ck)
            assert pk[0]["z"] == p0[0]["z"]
            assert pk[0]["Q"] == F32(p0[0]["Q"] * 2.0 ** -k)


def test_degenerate_units():
    # Reading R3: a zero unit gets Q = 1, z = 0 and recovers exactly to 0; a constant unit maps to
    # code 0 and recovers to within half a step of the constant.
    codes, p, sums = oracle.quantize(np.zeros((1, 7), F32))
    assert codes.tolist() == [[0] * 7] and p[0]["Q"] == 1.0 and p[0]["z"] == 0 and sums[0] == 0
    for c in (0.3, -2.5, 1e-8, -7e5):
        codes, p, _ = oracle.quantize(np.full((1, 5), c, F32))
        assert codes.max() == 0
        rec = oracle.recover(codes[0], p[0])
        assert np.all(np.abs(rec - F32(c)) <= 0.5 / p[0]["Q"] * (1 + 1e-6))
    # a range far narrower than the magnitude falls back to the degenerate rule
    v = np.array([[1000.0, np.nextafter(F32(1000.0), F32(2000.0))]], F32)
    codes, p, _ = oracle.quantize(v)
    assert p[0]["Q"] == F32(255.0) / F32(v.max())


def test_nonfinite_rejected():
    for bad in (np.nan, np.inf, -np.inf):
        v = np.array([[0.0, 1.0, bad, 2.0]], F32)
        with pytest.raises(oracle.OracleError) as e:
            oracle.quantize(v)
        assert e.value.status == oracle.ERR_NONFINITE


def test_per_row_matches_per_matrix_on_each_row():
    rng = np.random.Generator(np.random.PCG64(15))
    x = rng.normal(0, 1, (9, 33)).astype(F32)
    c_rows, p_rows, s_rows = oracle.quantize(x, oracle.PER_ROW)
    for r in range(9):
        c1, p1, s1 = oracle.quantize(x[r:r + 1], oracle.PER_MATRIX)
        assert np.array_equal(c1[0], c_rows[r]) and p1[0] == p_rows[r] and s1[0] == s_rows[r]
    c_mat, p_mat, _ = oracle.quantize(x, oracle.PER_MATRIX)
    assert p_mat[0]["vmin"] == x.min() and p_mat[0]["vmax"] == x.max()


# ------------------------------------------------------------------------------------------
# Integer product and recovery: eq. (1)
# ------------------------------------------------------------------------------------------

def _rand_operands(rng, M, N, K, ga):
    A = rng.normal(0.3, 1.0, (M, K)).astype(F32)
    W = rng.uniform(-0.1, 0.1, (N, K)).astype(F32)
    ca, pa, ra = oracle.quantize(A, ga)
    cw, pw, cs = oracle.quantize(W, oracle.PER_MATRIX)
    return A, W, ca, pa, ra, cw, pw, cs


@pytest.mark.parametrize("ga", [oracle.PER_MATRIX, oracle.PER_ROW])
def test_offset_product_equals_expanded_corrections(ga):
    # eq. (1): S = sum (a' + za)(w' + zw) = acc + zw * rowsum(a') + za * rowsum(w') + K za zw.
    rng = np.random.Generator(np.random.PCG64(16))
    for M, N, K in ((1, 1, 1), (3, 5, 7), (4, 9, 64), (2, 3, 129)):
        _, _, ca, pa, ra, cw, pw, cs = _rand_operands(rng, M, N, K, ga)
        out = oracle.qmatmul(ca, pa, ga, cw, pw)
        za = np.broadcast_to(pa["z"].astype(np.int64), (M,))[:, None]
        zw = np.int64(pw[0]["z"])
        expanded = out["acc"].astype(np.int64) + zw * ra.astype(np.int64)[:, None] \
            + za * cs.astype(np.int64)[None, :] + K * za * zw
        assert np.array_equal(out["S"], expanded)
        # raw accumulator: brute force over Python ints
        for m in range(M):
            for n in range(N):
                assert out["acc"][m, n] == sum(int(ca[m, k]) * int(cw[n, k]) for k in range(K))


def test_recovered_product_equals_product_of_recovered_values():
    # eq. (1) recovery 1/(Qa Qb) applied to S equals the fp64 inner product of eq. (3)-recovered
    # operands; and both are close to the fp32 product of the original values.
    rng = np.random.Generator(np.random.PCG64(17))
    M, N, K = 6, 10, 200
    A, W, ca, pa, _, cw, pw, _ = _rand_operands(rng, M, N, K, oracle.PER_ROW)
    out = oracle.qmatmul(ca, pa, oracle.PER_ROW, cw, pw)
    Qa = pa["Q"].astype(np.float64)[:, None]
    Qw = np.float64(pw[0]["Q"])
    ra = (ca.astype(np.float64) + pa["z"][:, None]) / Qa
    rw = (cw.astype(np.float64) + pw[0]["z"]) / Qw
    exact = ra @ rw.T
    y64 = out["S"].astype(np.float64) / (Qa * Qw)
    assert np.allclose(y64, exact, rtol=1e-12, atol=1e-12)
    # fp32 recovery: one conversion of S, one product of scales, one divide (3 roundings)
    assert np.all(np.abs(out["y"] - exact) <= 4 * 2.0 ** -24 * np.abs(exact) + 1e-30)
    # half-step bound against the unquantized product
    ea = 0.5 / Qa * (1 + 1e-4)
    ew = 0.5 / Qw * (1 + 1e-4)
    bound = (np.abs(A).astype(np.float64) @ np.full((K, N), ew)) + (ea * np.abs(W).sum(1)[None, :]) + K * ea * ew
    truth = A.astype(np.float64) @ W.astype(np.float64).T
    assert np.all(np.abs(out["y"] - truth) <= bound * 1.01)


def test_bias_added_after_recovery():
    # Fig. 1: y = R(Mult(Q(X), W')) + B.
    rng = np.random.Generator(np.random.PCG64(18))
    _, _, ca, pa, _, cw, pw, _ = _rand_operands(rng, 3, 4, 17, oracle.PER_ROW)
    b = rng.normal(0, 1, 4).astype(F32)
    y0 = oracle.qmatmul(ca, pa, oracle.PER_ROW, cw, pw)["y"]
    y1 = oracle.qmatmul(ca, pa, oracle.PER_ROW, cw, pw, bias=b)["y"]
    assert np.array_equal(y1, (y0 + b[None, :]).astype(F32))


def test_per_block_weight_params():
    # Weights quantized per gate matrix: n_blocks row blocks, each with its own (Q, z).
    rng = np.random.Generator(np.random.PCG64(19))
    K, Hh = 21, 5
    A = rng.normal(0, 1, (2, K)).astype(F32)
    ca, pa, _ = oracle.quantize(A, oracle.PER_ROW)
    blocks = [rng.uniform(-s, s, (Hh, K)).astype(F32) for s in (0.1, 0.5, 1.0, 2.0)]
    cws, pws = zip(*[oracle.quantize(b, oracle.PER_MATRIX)[:2] for b in blocks])
    cw = np.concatenate(cws)
    pw = np.concatenate(pws)
    y = oracle.qmatmul(ca, pa, oracle.PER_ROW, cw, pw, n_blocks=4)["y"]
    for g in range(4):
        yg = oracle.qmatmul(ca, pa, oracle.PER_ROW, cws[g], pws[g])["y"]
        assert np.array_equal(y[:, g * Hh:(g + 1) * Hh], yg)


def test_int32_accumulator_cannot_overflow_at_k_max():
    # 8-bit operands into 32-bit accumulators (Sec. 3.1): K * 255^2 <= 2^31 - 1 iff K <= 33025.
    assert oracle.K_MAX * 255 * 255 <= 2 ** 31 - 1 < (oracle.K_MAX + 1) * 255 * 255
    K = oracle.K_MAX
    ones = np.full((1, K), 255, np.uint8)
    p = np.zeros(1, oracle.QPARAMS_DTYPE)
    p[0] = (0.0, 1.0, 255.0, 0)
    out = oracle.qmatmul(ones, p, oracle.PER_MATRIX, ones, p)
    assert int(out["acc"][0, 0]) == K * 65025
    with pytest.raises(oracle.OracleError) as e:
        big = np.full((1, K + 1), 255, np.uint8)
        oracle.qmatmul(big, p, oracle.PER_MATRIX, big, p)
    assert e.value.status == oracle.ERR_K_TOO_LARGE


# ------------------------------------------------------------------------------------------
# Pinned transcendentals
# ------------------------------------------------------------------------------------------

def test_exp_within_two_ulp_of_libm():
    xs = np.concatenate([np.linspace(-87, 88, 40001), np.linspace(-1, 1, 4001), [0.0, -0.0, 1e-8, -1e-8]])
    xs = xs.astype(F32)
    e = np.array([oracle.exp_(float(x)) for x in xs], np.float64)
    ref = np.exp(xs.astype(np.float64))
    ulp = np.spacing(ref.astype(F32)).astype(np.float64)
    assert np.max(np.abs(e - ref) / ulp) <= 2.0
    assert oracle.exp_(0.0) == 1.0
    # clamping keeps results finite and normal
    assert oracle.exp_(1000.0) == oracle.exp_(88.0) and math.isfinite(oracle.exp_(1000.0))
    assert oracle.exp_(-1000.0) == oracle.exp_(-87.0) > 1.17549435e-38


def test_sigmoid_tanh_against_libm():
    xs = np.linspace(-30, 30, 20001).astype(F32)
    s = np.array([oracle.sigmoid(float(x)) for x in xs])
    t = np.array([oracle.tanh(float(x)) for x in xs])
    x64 = xs.astype(np.float64)
    assert np.max(np.abs(s - 1 / (1 + np.exp(-x64)))) <= 2e-7
    assert np.max(np.abs(t - np.tanh(x64))) <= 3e-7
    assert oracle.tanh(0.0) == 0.0 and oracle.sigmoid(0.0) == 0.5


# ------------------------------------------------------------------------------------------
# LSTM stack: textbook reduction and structural invariants
# ------------------------------------------------------------------------------------------

def _unpack(wl, params):
    """Split the packed parameters (layout documented in inputs.LstmWorkload.make_params)."""
    H, P, R = wl.hidden, wl.proj, wl.R
    off = 0
    layers = []

    def take(n, shape):
        nonlocal off
        a = params[off:off + n].reshape(shape)
        off += n
        return a

    for l in range(wl.num_layers):
        Ik = wl.layer_in(l)
        wx = take(4 * H * Ik, (4, H, Ik))
        wh = take(4 * H * R, (4, H, R))
        b = take(4 * H, (4, H))
        wp = take(P * H, (P, H)) if P > 0 else None
        layers.append((wx, wh, b, wp))
    out = None
    if wl.num_classes > 0:
        wo = take(wl.num_classes * R, (wl.num_classes, R))
        bo = take(wl.num_classes, (wl.num_classes,))
        out = (wo, bo)
    assert off == params.size
    return layers, out


def _recovered_row(v):
    c, p, _ = oracle.quantize(np.asarray(v, F32)[None, :], oracle.PER_ROW)
    return (c[0].astype(np.float64) + int(p[0]["z"])) / float(p[0]["Q"])


def _recovered_mat(w, nb=1):
    """eq. (3) recovery of a weight matrix quantized as nb row blocks, each its own unit."""
    out = []
    for blk in np.split(np.asarray(w, F32), nb):
        c, p, _ = oracle.quantize(blk, oracle.PER_MATRIX)
        out.append((c.astype(np.float64) + int(p[0]["z"])) / float(p[0]["Q"]))
    return np.concatenate(out)


def _sig(x):
    return 1.0 / (1.0 + np.exp(-x))


def _textbook_check(wl, params, x, res, tol_h, nb=1):
    """Teacher-forced: every step of the oracle's LSTM equals a float64 textbook LSTM step (no
    peepholes, gates [i, f, g, o]) applied to eq. (3)-recovered inputs and weights, fed with the
    oracle's own previous outputs."""
    layers, out = _unpack(wl, params)
    B, T, _ = x.shape
    H = wl.hidden
    worst = 0.0
    for l, (wx, wh, b, wp) in enumerate(layers):
        rwx = np.stack([_recovered_mat(wx[g], nb) for g in range(4)])
        rwh = np.stack([_recovered_mat(wh[g], nb) for g in range(4)])
        rwp = _recovered_mat(wp, nb) if wp is not None else None
        for bb in range(B):
            c = np.zeros(H)
            hprev = np.zeros(wl.R, F32)
            for t in range(T):
                xin = x[bb, t] if l == 0 else res["h_all"][l - 1, bb, t]
                rx = _recovered_row(xin)
                rh = _recovered_row(hprev)
                pre = np.einsum("ghk,k->gh", rwx, rx) + b.astype(np.float64) + np.einsum("ghk,k->gh", rwh, rh)
                i, f, g, o = _sig(pre[0]), _sig(pre[1]), np.tanh(pre[2]), _sig(pre[3])
                c = f * c + i * g
                m = o * np.tanh(c)
                h = rwp @ _recovered_row(m.astype(F32)) if rwp is not None else m
                got = res["h_all"][l, bb, t].astype(np.float64)
                worst = max(worst, float(np.max(np.abs(got - h))))
                hprev = res["h_all"][l, bb, t]
    assert worst <= tol_h, worst
    if out is not None and wl.output_mode == oracle.OUT_QUANT:
        wo, bo = out
        rwo = _recovered_mat(wo, nb)
        for bb in range(B):
            for t in range(T):
                r = _recovered_row(res["h_all"][-1, bb, t])
                lg = rwo @ r + bo
                assert np.max(np.abs(res["logits"][bb, t] - lg)) <= 1e-5 * (1 + np.abs(lg).max())
                e = np.exp(lg - lg.max())
                assert np.max(np.abs(res["y"][bb, t] - e / e.sum())) <= 1e-6


def _small(name="t", L=2, I=7, H=9, P=0, C=0, B=2, T=6, seed=5, mode=None, fb=1.0):
    return inputs.LstmWorkload(name, seed=seed, num_layers=L, input_dim=I, hidden=H, proj=P, num_classes=C,
                               batch=B, frames=T, w_range=0.5, forget_bias=fb,
                               output_mode=(mode if mode is not None else (1 if C > 0 else 0)))


def _run(wl, params, x, nb=0, **kw):
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode, nb)
    return oracle.lstm_forward(d, params, x, want_h_all=True, want_logits=wl.num_classes > 0, **kw)


@pytest.mark.parametrize("cfg", [dict(), dict(L=1, I=3, H=4, B=1, T=9), dict(L=3, H=16, C=11),
                                 dict(L=2, H=12, C=5, fb=0.0)])
def test_lstm_reduces_to_textbook_lstm_on_recovered_operands(cfg):
    wl = _small(**cfg)
    params, x = wl.make()
    res = _run(wl, params, x)
    _textbook_check(wl, params, x, res, tol_h=2e-6)


# a projection narrower than the cells, and one wider than both the cells and the input (the
# recurrent input is then the widest row a step quantizes)
@pytest.mark.parametrize("cfg", [dict(L=2, I=6, H=10, P=4, C=7, B=2, T=5), dict(L=2, I=5, H=6, P=20, C=7, B=2, T=5)])
def test_lstmp_reduces_to_textbook_on_recovered_operands(cfg):
    wl = _small(**cfg)
    params, x = wl.make()
    res = _run(wl, params, x)
    # the projection re-quantizes m, computed here in fp64: a code may flip on an fp32 tie
    _textbook_check(wl, params, x, res, tol_h=2e-3)


def test_lstm_scalar_case_is_the_float_lstm():
    # One input, one cell: every unit has a single value, so the degenerate rule (R3) recovers it
    # to within a few ulp and the quantized LSTM equals the float LSTM (no quantization loss).
    wl = _small(L=1, I=1, H=1, B=1, T=20, fb=0.0)
    params, x = wl.make()
    res = _run(wl, params, x)
    wx, wh, b, _ = _unpack(wl, params)[0][0]
    c = 0.0
    h = 0.0
    for t in range(20):
        pre = wx[:, 0, 0].astype(np.float64) * float(x[0, t, 0]) + b[:, 0] + wh[:, 0, 0].astype(np.float64) * h
        i, f, g, o = _sig(pre[0]), _sig(pre[1]), math.tanh(pre[2]), _sig(pre[3])
        c = f * c + i * g
        h = o * math.tanh(c)
        assert abs(float(res["h_all"][0, 0, t, 0]) - h) <= 2e-6
        h = float(res["h_all"][0, 0, t, 0])


def test_quantized_lstm_close_to_float_lstm():
    # 'mismatch' vs 'match' (Sec. 5): post-training 8-bit quantization perturbs the float model
    # only slightly. A swapped gate or a wrong offset produces O(1) differences instead.
    wl = inputs.SMALL_1x128
    params, x = wl.make(frames=40)
    res = _run(wl, params, x)
    wx, wh, b, _ = _unpack(wl, params)[0][0]
    c = np.zeros(wl.hidden)
    h = np.zeros(wl.hidden)
    diffs = []
    for t in range(40):
        pre = np.einsum("ghk,k->gh", wx.astype(np.float64), x[0, t]) + b + np.einsum("ghk,k->gh", wh, h)
        c = _sig(pre[1]) * c + _sig(pre[0]) * np.tanh(pre[2])
        h = _sig(pre[3]) * np.tanh(c)
        diffs.append(np.abs(res["h_all"][0, 0, t] - h))
    diffs = np.array(diffs)
    assert diffs.max() < 0.03 and diffs.mean() < 0.004


def test_batch_independence_and_streaming_state():
    wl = _small(L=3, H=8, C=6, B=3, T=10)
    params, x = wl.make()
    full = _run(wl, params, x)
    for b in range(3):
        one = _run(wl, params, x[b:b + 1])
        assert np.array_equal(one["y"][0], full["y"][b])
        assert np.array_equal(one["h"][:, 0], full["h"][:, b])
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes)
    a = oracle.lstm_forward(d, params, x[:, :4])
    b2 = oracle.lstm_forward(d, params, x[:, 4:], h0=a["h"], c0=a["c"])
    assert np.array_equal(np.concatenate([a["y"], b2["y"]], 1), full["y"])
    assert np.array_equal(b2["h"], full["h"]) and np.array_equal(b2["c"], full["c"])


def test_input_permutation_invariance():
    # Integer sums and per-row ranges do not depend on the order of the K inputs.
    wl = _small(L=2, I=9, H=6, C=4, B=2, T=5)
    params, x = wl.make()
    base = _run(wl, params, x)
    perm = np.random.Generator(np.random.PCG64(20)).permutation(wl.input_dim)
    layers, _ = _unpack(wl, params)
    p2 = params.copy()
    wx = layers[0][0]
    p2[:wx.size] = wx[:, :, perm].ravel()
    res = _run(wl, p2, np.ascontiguousarray(x[:, :, perm]))
    assert np.array_equal(res["y"], base["y"])


def test_softmax_rows():
    wl = _small(L=1, H=6, C=13, B=2, T=4)
    params, x = wl.make()
    res = _run(wl, params, x)
    assert np.allclose(res["y"].sum(-1), 1.0, atol=2e-6)
    lg = res["logits"].astype(np.float64)
    e = np.exp(lg - lg.max(-1, keepdims=True))
    assert np.max(np.abs(res["y"] - e / e.sum(-1, keepdims=True))) <= 1e-6


def test_softmax_of_many_nearly_equal_logits():
    # 8192 classes whose logits lie within +-5e-4 (a wide output layer with small weights): every
    # posterior equals the fp64 softmax of the same logits to within the pinned E's error (a few
    # fp32 ulp), which a running fp32 sum of the 8192 nearly equal terms misses by far
    wl = inputs.LstmWorkload("flat", seed=3, num_layers=1, input_dim=5, hidden=8, proj=0, num_classes=8192,
                             batch=1, frames=3, w_range=0.5, out_w_range=2e-4)
    params, x = wl.make()
    res = _run(wl, params, x)
    lg = res["logits"].astype(np.float64)
    assert np.abs(lg).max() < 1e-3
    e = np.exp(lg - lg.max(-1, keepdims=True))
    want = e / e.sum(-1, keepdims=True)
    assert np.max(np.abs(res["y"] / want - 1.0)) <= 5e-7
    # the same terms summed in a running fp32 sum drift by more than 1e-5 of the posterior
    ef = np.array([oracle.exp_(float(v)) for v in (res["logits"][0, 0] - res["logits"][0, 0].max())], np.float32)
    s = np.float32(0.0)
    for v in ef:
        s = np.float32(s + v)
    assert abs(float(s) / ef.astype(np.float64).sum() - 1.0) > 1e-5


def test_float_output_layer_variant():
    # 'quant' (Sec. 5): every layer quantized except the softmax layer, which stays float.
    wl = _small(L=2, H=8, C=9, B=1, T=5, mode=2)
    params, x = wl.make()
    res = _run(wl, params, x)
    _, (wo, bo) = _unpack(wl, params)
    lg = res["h_all"][-1, 0].astype(np.float64) @ wo.T.astype(np.float64) + bo
    assert np.max(np.abs(res["logits"][0] - lg)) <= 1e-6
    wl_q = _small(L=2, H=8, C=9, B=1, T=5, mode=1)
    resq = _run(wl_q, params, x)
    assert np.array_equal(resq["h_all"], res["h_all"])  # layers below the output are identical


def test_weight_quantization_units():
    wl = _small(L=2, I=5, H=6, P=3, C=4)
    params, _ = wl.make()
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes)
    codes, qp = oracle.lstm_quantize_weights(d, params)
    assert len(qp) == 2 * 9 + 1  # 4 Wx + 4 Wh + Wp per layer, then Wo
    layers, (wo, _) = _unpack(wl, params)
    c0, p0, _ = oracle.quantize(layers[0][0][2], oracle.PER_MATRIX)  # layer 0, Wx gate g
    off = 2 * wl.hidden * wl.input_dim
    assert np.array_equal(codes[off:off + c0.size].reshape(c0.shape), c0) and qp[2] == p0[0]


# ------------------------------------------------------------------------------------------
# Frozen oracle outputs (tests/golden/make_golden.py writes them from the oracle alone)
# ------------------------------------------------------------------------------------------

def test_golden_fixtures_unchanged():
    import json
    import os
    here = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
    g = json.load(open(os.path.join(here, "oracle_quantizer_rows.json")))
    x = np.array([float.fromhex(v) for v in g["x_hex"]], F32).reshape(g["rows"], g["cols"])
    codes, p, sums = oracle.quantize(x, oracle.PER_ROW)
    assert codes.ravel().tolist() == g["codes"] and sums.tolist() == g["sums"] and p["z"].tolist() == g["z"]
    assert [float(v).hex() for v in p["Q"]] == g["Q_hex"]
    g = json.load(open(os.path.join(here, "oracle_lstm_tiny.json")))
    wl = inputs.LstmWorkload(g["workload"], seed=g["seed"], num_layers=g["num_layers"], input_dim=g["input_dim"],
                             hidden=g["hidden"], proj=0, num_classes=g["num_classes"], batch=g["batch"],
                             frames=g["frames"], w_range=g["w_range"], forget_bias=g["forget_bias"])
    params, x = wl.make()
    res = oracle.lstm_forward(oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, 0, wl.num_classes), params, x)
    assert [float(v).hex() for v in res["y"].ravel()] == g["y_hex"]
    assert [float(v).hex() for v in res["h"].ravel()] == g["h_hex"]


# ------------------------------------------------------------------------------------------
# Frame stacking (Sec. 4 frontend; reading R9 for the sequence end)
# ------------------------------------------------------------------------------------------

def _stack_reference(x, n, stride):
    """The same definition by array slicing: pad the end by repeating the last frame, take n
    shifted views, concatenate along features, keep every stride-th."""
    B, T, I = x.shape
    padded = np.concatenate([x, np.repeat(x[:, -1:], n - 1, axis=1)], axis=1)
    windows = np.concatenate([padded[:, k:k + T] for k in range(n)], axis=2)
    return windows[:, ::stride]


def test_stack_frames_identity_and_subsampling():
    g = np.random.Generator(np.random.PCG64(21))
    x = g.normal(0, 1, (3, 11, 5)).astype(np.float32)
    assert np.array_equal(oracle.stack_frames(x, 1, 1), x)
    assert np.array_equal(oracle.stack_frames(x, 1, 3), x[:, ::3])


@pytest.mark.parametrize("n,stride,T", [(8, 3, 300), (8, 3, 7), (8, 3, 1), (3, 2, 10), (5, 1, 4), (2, 7, 20)])
def test_stack_frames_matches_sliced_windows(n, stride, T):
    g = np.random.Generator(np.random.PCG64(n * 100 + stride * 10 + T))
    x = g.normal(0, 1, (2, T, 6)).astype(np.float32)
    got = oracle.stack_frames(x, n, stride)
    assert got.shape == (2, -(-T // stride), n * 6)
    assert np.array_equal(got, _stack_reference(x, n, stride))


def test_stack_frames_paper_frontend():
    """40-dim frames, 8 stacked (7 of right context), every third presented: 320 features per input,
    one input per 30 ms of 10 ms frames (T = 300 frames -> 100 inputs)."""
    x = np.arange(1 * 300 * 40, dtype=np.float32).reshape(1, 300, 40)
    s = oracle.stack_frames(x, 8, 3)
    assert s.shape == (1, 100, 320)
    for t in (0, 1, 50, 97):
        for k in range(8):
            assert np.array_equal(s[0, t, 40 * k:40 * (k + 1)], x[0, 3 * t + k])
    # the last input reaches past frame 299: frames 297..304 -> 297, 298, 299, 299, ...
    last = s[0, 99].reshape(8, 40)[:, 0] / 40
    assert list(last) == [297, 298, 299, 299, 299, 299, 299, 299]



# ------------------------------------------------------------------------------------------
# Sub-matrix granularity (Sec. 3.1): a weight matrix quantized as row blocks, each its own unit
# ------------------------------------------------------------------------------------------

def _heterogeneous_blocks(wl, params, nb, seed=3):
    """Rescale the row blocks of every weight matrix by very different factors (the case finer
    granularity is for)."""
    layers, out = _unpack(wl, params)
    p = params.copy()
    f = np.random.Generator(np.random.PCG64(seed)).choice([0.05, 0.3, 1.0, 4.0], size=nb)
    scale = lambda w: (w.reshape(nb, -1) * f[:, None]).reshape(w.shape)
    chunks = []
    for wx, wh, b, wp in layers:
        chunks += [np.stack([scale(wx[g]) for g in range(4)]).ravel(),
                   np.stack([scale(wh[g]) for g in range(4)]).ravel(), b.ravel()]
        if wp is not None:
            chunks.append(scale(wp).ravel())
    if out is not None:
        chunks += [scale(out[0]).ravel(), out[1].ravel()]
    return np.concatenate(chunks).astype(F32)


@pytest.mark.parametrize("cfg,nb", [(dict(L=2, I=7, H=12, C=6), 3), (dict(L=2, I=6, H=16, P=8, C=8, T=5), 4),
                                    (dict(L=1, I=5, H=6, B=1, T=8), 6)])
def test_sub_matrix_units_reduce_to_textbook(cfg, nb):
    """With nb units per matrix the oracle's LSTM is the textbook LSTM on operands recovered block
    by block; using another block's parameters would break this by the ratio of their scales."""
    wl = _small(**cfg)
    params, x = wl.make()
    params = _heterogeneous_blocks(wl, params, nb)
    res = _run(wl, params, x, nb=nb)
    _textbook_check(wl, params, x, res, tol_h=2e-3 if wl.proj else 2e-6, nb=nb)


def test_sub_matrix_units_are_more_precise():
    """Sec. 3.1: subdividing a matrix into individually quantized sub-matrices gives better
    precision: the recovered weights of blocks with very different scales are closer to the
    float weights, block by block, and so is the quantized LSTM to the float LSTM."""
    wl = _small(L=1, I=16, H=32, B=1, T=30)
    params, x = wl.make()
    params = _heterogeneous_blocks(wl, params, 4)
    wx = _unpack(wl, params)[0][0][0]
    for g in range(4):
        e1 = np.abs(_recovered_mat(wx[g], 1) - wx[g]).max(axis=1)
        e4 = np.abs(_recovered_mat(wx[g], 4) - wx[g]).max(axis=1)
        assert np.all(e4 <= e1 * (1 + 1e-6))
    one, four = _run(wl, params, x, nb=1), _run(wl, params, x, nb=4)
    float_h = _run(wl, params, x, nb=32)  # one unit per row: closest to float
    d1 = np.abs(one["h_all"] - float_h["h_all"]).mean()
    d4 = np.abs(four["h_all"] - float_h["h_all"]).mean()
    assert d4 < d1


def test_sub_matrix_weight_codes_by_block():
    wl = _small(L=2, I=5, H=8, P=4, C=4)
    params, _ = wl.make()
    d = oracle.desc(2, 5, 8, 4, 4, oracle.OUT_QUANT, 2)
    codes, prm = oracle.lstm_quantize_weights(d, params)
    assert len(prm) == 2 * (9 * 2 + 1)
    wx0 = _unpack(wl, params)[0][0][0][0]  # first gate matrix of layer 0: two units of 4 rows
    for blk in range(2):
        c, p, _ = oracle.quantize(wx0[4 * blk:4 * blk + 4], oracle.PER_MATRIX)
        assert np.array_equal(codes[4 * blk * 5:(4 * blk + 4) * 5].reshape(4, 5), c)
        assert prm[blk]["Q"] == p[0]["Q"] and prm[blk]["z"] == p[0]["z"]
    assert oracle.lstm_param_count(d) == params.size
    bad = oracle.desc(1, 5, 9, 0, 0, oracle.OUT_NONE, 2)  # 9 rows do not split in 2
    with pytest.raises(oracle.OracleError):
        oracle.lstm_forward(bad, np.zeros(oracle.lstm_param_count(bad), F32), np.zeros((1, 1, 5), F32))
