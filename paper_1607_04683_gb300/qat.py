"""Quantization-aware training step of Algorithm 1 (Sec. 3.2) for fully connected layers.

Forward pass: infer-and-recover. The layer computes what inference computes (Sec. 3.1): the
full-precision weights are quantized (quantize(w), one unit per weight matrix or per block of
rows), the layer input is quantized on the fly (one unit per row), the integer product with the
offset terms of eq. (1) runs on the device and is recovered by eq. (3), and the float bias is
added. Every one of those steps runs in libqnn's kernels (qnn_quantize, qnn_qmatmul).

Backward pass: full precision, as Algorithm 1 prescribes. The error propagates through the
full-precision weights (error()), the weight gradient pairs the error with the layer's input as it
came out of the quantized forward pass (wgradient()), and the bias gradient sums the error
(bgradient()). No quantization term enters the gradients; the optimizer updates the
full-precision parameters, which are quantized again at the next forward pass.

"quant-all" trains with every layer quantized, "quant" with every layer but the softmax layer
(Sec. 5): a network built from QuantLinear layers and a plain float output layer is the latter.
"""
from __future__ import annotations

import torch

from . import qnn


def quantize_weights(w: torch.Tensor, n_blocks: int = 1):
    """quantize(w) of Algorithm 1: w [N, K] fp32 CUDA, n_blocks equal row blocks each one unit
    (Sec. 3.1 granularity). Returns (codes u8 [N, K], params [n_blocks], row code sums [N])."""
    N = w.shape[0]
    if n_blocks < 1 or N % n_blocks:
        raise ValueError("n_blocks must divide the number of rows")
    per = N // n_blocks
    parts = [qnn.qnn_quantize(w[b * per:(b + 1) * per].contiguous(), qnn.PER_MATRIX) for b in range(n_blocks)]
    if n_blocks == 1:
        return parts[0]
    return (torch.cat([p[0] for p in parts]), torch.cat([p[1] for p in parts]), torch.cat([p[2] for p in parts]))


def infer_and_recover(x: torch.Tensor, w: torch.Tensor, b: torch.Tensor | None, n_blocks: int = 1) -> torch.Tensor:
    """The quantized layer of Sec. 3.1 on x [M, K]: R(Q(x) quantize(w)^T) + b, fp32 [M, N]."""
    cw, pw, cs = quantize_weights(w, n_blocks)
    ca, pa, ra = qnn.qnn_quantize(x, qnn.PER_ROW)
    y, _ = qnn.qnn_qmatmul(ca, pa, qnn.PER_ROW, ra, cw, pw, cs, n_blocks=n_blocks,
                           bias=None if b is None else b.detach().contiguous())
    return y


class _QuantizedLinear(torch.autograd.Function):
    @staticmethod
    def forward(ctx, x, w, b, n_blocks):
        x2 = x.reshape(-1, x.shape[-1]).contiguous()
        ctx.save_for_backward(x2, w)
        ctx.has_bias = b is not None
        ctx.in_shape = x.shape
        y = infer_and_recover(x2.detach(), w.detach().contiguous(), b, n_blocks)
        return y.reshape(*x.shape[:-1], w.shape[0])

    @staticmethod
    def backward(ctx, gy):
        x2, w = ctx.saved_tensors
        g = gy.reshape(-1, w.shape[0])
        gx = (g @ w).reshape(ctx.in_shape) if ctx.needs_input_grad[0] else None  # error()
        gw = g.t() @ x2 if ctx.needs_input_grad[1] else None                       # wgradient()
        gb = g.sum(0) if ctx.has_bias and ctx.needs_input_grad[2] else None         # bgradient()
        return gx, gw, gb, None


class QuantLinear(torch.nn.Module):
    """A fully connected layer trained by Algorithm 1: quantized forward, full-precision backward."""

    def __init__(self, in_features: int, out_features: int, bias: bool = True, n_blocks: int = 1,
                 device="cuda"):
        super().__init__()
        self.weight = torch.nn.Parameter(torch.empty(out_features, in_features, device=device))
        self.bias = torch.nn.Parameter(torch.zeros(out_features, device=device)) if bias else None
        self.n_blocks = n_blocks
        torch.nn.init.uniform_(self.weight, -1.0 / in_features ** 0.5, 1.0 / in_features ** 0.5)

    def forward(self, x):
        return _QuantizedLinear.apply(x, self.weight, self.bias, self.n_blocks)
