"""The GPU parity rules (tests/parity.py) can fail where they must, on the CPU.

Mutation checks on oracle outputs of the 5 x 500-cell, 2000-class model, whose posteriors all lie
within a few percent of 1/C: one logit moved by 0.01, an output layer that returns zero logits,
and one posterior scaled by 1 + 1e-4 each fail the comparison, while a softmax whose sum runs in
another order (what the GPU does) passes it.
"""
import numpy as np
import pytest

import oracle
import parity
from paper_1607_04683_gb300 import inputs


@pytest.fixture(scope="module")
def ref():
    wl = inputs.LSTM_5x500_B1
    params, x = wl.make(frames=4)
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    out = oracle.lstm_forward(d, params, x, want_h_all=True, want_logits=True)
    out["wl"] = wl
    return out


def _softmax_pairwise(logits):
    """fp32 softmax with the pinned exponential and a pairwise (tree) sum: another summation order."""
    lg = np.asarray(logits, np.float32)
    mx = lg.max(-1, keepdims=True)
    e = np.vectorize(oracle.exp_, otypes=[np.float32])(lg - mx).astype(np.float32)
    s = e.copy()
    while s.shape[-1] > 1:
        if s.shape[-1] % 2:
            s = np.concatenate([s, np.zeros(s.shape[:-1] + (1,), np.float32)], -1)
        s = (s[..., 0::2] + s[..., 1::2]).astype(np.float32)
    return (e / s).astype(np.float32)


def _copy(r):
    return {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in r.items()}


def test_posteriors_are_near_uniform_here(ref):
    # the case the absolute bar alone cannot see: every posterior within 4% of 1/C
    C = ref["wl"].num_classes
    assert np.all(np.abs(ref["y"] * C - 1.0) < 0.04)


def test_identical_outputs_pass(ref):
    wl = ref["wl"]
    parity.compare(_copy(ref), ref, wl.num_layers, wl.num_classes, 1)


def test_another_summation_order_passes(ref):
    y = _softmax_pairwise(ref["logits"][0, :2])
    parity.check_posteriors(y, ref["y"][0, :2])


def test_one_logit_moved_by_a_hundredth_fails(ref):
    wl = ref["wl"]
    got = _copy(ref)
    got["logits"][0, 1, 5] += np.float32(0.01)
    with pytest.raises(AssertionError):
        parity.check_logits(got["logits"], ref["logits"], 1)
    got["y"][0, 1] = _softmax_pairwise(got["logits"][0, 1:2])[0]
    with pytest.raises(AssertionError):
        parity.check_posteriors(got["y"], ref["y"])
    with pytest.raises(AssertionError):
        parity.compare(got, ref, wl.num_layers, wl.num_classes, 1)


def test_zero_logits_fail(ref):
    got = _copy(ref)
    got["logits"][:] = 0.0
    got["y"][:] = np.float32(1.0 / ref["wl"].num_classes)
    assert np.max(np.abs(got["y"] - ref["y"])) <= parity.POSTERIOR_ABS  # the absolute bar alone passes
    with pytest.raises(AssertionError):
        parity.check_posteriors(got["y"], ref["y"])
    with pytest.raises(AssertionError):
        parity.check_logits(got["logits"], ref["logits"], 1)


def test_one_posterior_off_by_1e4_relative_fails(ref):
    got = _copy(ref)
    got["y"][0, 2, 77] *= np.float32(1.0 + 1e-4)
    with pytest.raises(AssertionError):
        parity.check_posteriors(got["y"], ref["y"])


def test_float_logit_bound_catches_a_dropped_term():
    # the float output layer's bound (K u sum |r w|) is far below a dropped product term
    r = np.random.Generator(np.random.PCG64(9))
    top = r.uniform(-1, 1, (3, 40)).astype(np.float32)
    w = r.uniform(-0.5, 0.5, (7, 40)).astype(np.float32)
    exact = (top.astype(np.float64) @ w.astype(np.float64).T).astype(np.float32)
    fp32 = np.zeros((3, 7), np.float32)
    for k in range(40):
        fp32 = (fp32 + top[:, k:k + 1] * w[:, k]).astype(np.float32)
    parity.check_logits(fp32, exact, 2, top, w)
    dropped = (fp32 - top[:, 13:14] * w[:, 13]).astype(np.float32)
    with pytest.raises(AssertionError):
        parity.check_logits(dropped, exact, 2, top, w)
