"""Comparison rules of the GPU parity tests (imported by the test modules; no GPU needed).

The bar, per output of qnn_lstm_forward:
  - every layer output h_t, the final state (h, c) and, for the 8-bit output layer ("quant-all",
    Sec. 5), the logits: bit-exact. Both sides run the same fp32 operations in the same order
    (eq. 1 in exact integers, eq. 3's recovery, the bias add of Fig. 1), so any difference is a bug.
  - logits of the float output layer ("quant"): the oracle sums in fp64 and rounds once, the GPU
    sums K products in fp32; the bound is the fp32 dot-product error K u sum_k |r_k w_k| plus the
    rounding of the bias add (u = 2^-24).
  - posteriors: within 1e-4 absolute AND 1e-5 relative (+1e-12) element by element. Given equal
    logits, E(l - max) is the same on both sides; only the softmax sum's order differs (a
    sequential fp32 sum of C <= 8192 positive terms is within a few 1e-6 of any other order).
The relative half matters: at the configured model sizes every posterior lies within a few percent
of 1/C, so an absolute 1e-4 alone would accept an output layer that returned all-zero logits.
"""
import numpy as np

POSTERIOR_ABS = 1e-4
POSTERIOR_REL = 1e-5
U32 = 2.0 ** -24


def check_posteriors(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape
    d = np.abs(got - ref)
    assert np.all(d <= POSTERIOR_ABS), f"posteriors: max abs diff {d.max():.3g}"
    rel_ok = d <= POSTERIOR_REL * np.abs(ref) + 1e-12
    assert np.all(rel_ok), f"posteriors: max rel diff {np.max(d / (np.abs(ref) + 1e-30)):.3g}"


def float_logit_bound(top, w_out, ref_logits):
    """Error bound of fp32 logits = sum_k r_k w_k + b against the once-rounded fp64 value: the
    top layer's outputs top [..., K] (bit-exact on both sides) and the output weights w_out [C, K]."""
    K = top.shape[-1]
    absdot = np.abs(top.astype(np.float64)) @ np.abs(w_out.astype(np.float64)).T
    return (K + 2) * U32 * absdot + 2 * U32 * np.abs(ref_logits.astype(np.float64))


def check_logits(got, ref, output_mode, top=None, w_out=None):
    got = np.asarray(got, np.float32)
    ref = np.asarray(ref, np.float32)
    assert got.shape == ref.shape
    if output_mode == 1:
        assert np.array_equal(got.view(np.uint32), ref.view(np.uint32)), \
            f"8-bit output layer logits differ: max diff {np.max(np.abs(got - ref)):.3g}"
    else:
        bound = float_logit_bound(top, w_out, ref)
        d = np.abs(got.astype(np.float64) - ref.astype(np.float64))
        assert np.all(d <= bound), f"float output layer logits beyond the fp32 dot-product bound: {d.max():.3g}"


def compare(got, ref, num_layers, num_classes, output_mode=1, w_out=None):
    """got / ref: dicts with y, h, c and optionally h_all, logits (ref from the oracle)."""
    if "h_all" in got and "h_all" in ref:
        for l in range(num_layers):
            assert np.array_equal(got["h_all"][l], ref["h_all"][l]), f"layer {l} outputs differ"
    assert np.array_equal(got["h"], ref["h"]) and np.array_equal(got["c"], ref["c"])
    if num_classes > 0:
        if "logits" in got and "logits" in ref:
            top = ref["h_all"][num_layers - 1] if "h_all" in ref else None
            check_logits(got["logits"], ref["logits"], output_mode, top, w_out)
        check_posteriors(got["y"], ref["y"])
    else:
        assert np.array_equal(got["y"], ref["y"])
