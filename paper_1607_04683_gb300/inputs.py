"""Seeded synthetic inputs shared by the tests, the benchmark and the oracle checks.

This module holds no arithmetic of the method: it only draws fp32 numbers and lays them out in the
packed parameter order that the library and the oracle both accept. The paper's features and
trained models are proprietary (Sec. 4); these shapes and value ranges stand in for them:
LSTM stacks of 4-5 layers of 300-500 cells, optional recurrent projections, 40-dimensional
log-mel frames (Sec. 4), and an 8-bit softmax output layer ("quant-all", Sec. 5).

Generator: numpy ``Generator(PCG64(seed))``; float64 draws cast to fp32. Draw order for a model:
for each layer, for each gate in [i, f, g, o]: Wx[g] then Wh[g]; then Wp (projection, if any);
after all layers Wo (if any); then the frames x in [B, T, I] order (per-sequence mean offsets,
when used, are drawn just before x). Biases are deterministic (0, or 1.0 on the forget gate).
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

GATES = ("i", "f", "g", "o")


@dataclass(frozen=True)
class LstmWorkload:
    name: str
    seed: int
    num_layers: int
    input_dim: int
    hidden: int
    proj: int
    num_classes: int
    batch: int
    frames: int
    w_range: float
    forget_bias: float = 0.0
    seq_mean_range: float = 0.0  # per-sequence mean offset ~ U(-r, r) added to x
    output_mode: int = 1  # 0 none, 1 quantized output layer ("quant-all"), 2 float output layer ("quant")
    out_w_range: float = 0.0  # output weights ~ U(-r, r) if r > 0 (spreads the logits), else w_range

    @property
    def R(self) -> int:
        return self.proj if self.proj > 0 else self.hidden

    def layer_in(self, l: int) -> int:
        return self.input_dim if l == 0 else self.R

    def param_count(self) -> int:
        H, P, R = self.hidden, self.proj, self.R
        n = 0
        for l in range(self.num_layers):
            n += 4 * H * self.layer_in(l) + 4 * H * R + 4 * H + (P * H if P > 0 else 0)
        if self.num_classes > 0:
            n += self.num_classes * R + self.num_classes
        return n

    def make_params(self, rng: np.random.Generator) -> np.ndarray:
        """Packed fp32 parameters: per layer Wx[4][H][Ik], Wh[4][H][R], b[4][H], Wp[P][H];
        then Wo[C][R], bo[C]."""
        H, P, R, a = self.hidden, self.proj, self.R, self.w_range
        out = np.empty(self.param_count(), np.float32)
        off = 0
        for l in range(self.num_layers):
            Ik = self.layer_in(l)
            wx = np.empty((4, H, Ik), np.float32)
            wh = np.empty((4, H, R), np.float32)
            for g in range(4):
                wx[g] = rng.uniform(-a, a, (H, Ik)).astype(np.float32)
                wh[g] = rng.uniform(-a, a, (H, R)).astype(np.float32)
            b = np.zeros((4, H), np.float32)
            b[1] = self.forget_bias
            for arr in (wx, wh, b):
                out[off:off + arr.size] = arr.ravel()
                off += arr.size
            if P > 0:
                wp = rng.uniform(-a, a, (P, H)).astype(np.float32)
                out[off:off + wp.size] = wp.ravel()
                off += wp.size
        if self.num_classes > 0:
            ao = self.out_w_range if self.out_w_range > 0 else a
            wo = rng.uniform(-ao, ao, (self.num_classes, R)).astype(np.float32)
            out[off:off + wo.size] = wo.ravel()
            off += wo.size
            out[off:off + self.num_classes] = 0.0
            off += self.num_classes
        assert off == out.size
        return out

    def out_weights(self, params: np.ndarray) -> np.ndarray:
        """The output layer's weights Wo [C, R] inside a packed parameter buffer."""
        C, R = self.num_classes, self.R
        return params[params.size - C * R - C: params.size - C].reshape(C, R)

    def make_frames(self, rng: np.random.Generator, batch: int | None = None, frames: int | None = None) -> np.ndarray:
        B = self.batch if batch is None else batch
        T = self.frames if frames is None else frames
        mu = None
        if self.seq_mean_range > 0:
            mu = rng.uniform(-self.seq_mean_range, self.seq_mean_range, B)
        x = rng.standard_normal((B, T, self.input_dim))
        if mu is not None:
            x = x + mu[:, None, None]
        return x.astype(np.float32)

    def make(self, batch: int | None = None, frames: int | None = None):
        rng = np.random.Generator(np.random.PCG64(self.seed))
        params = self.make_params(rng)
        x = self.make_frames(rng, batch, frames)
        return params, x


# The workloads: shapes follow the paper's model family (Sec. 4: 4-5 layers of N = 300..500 cells,
# projections of P units after each layer) and an embedded acoustic model's frame rate; the last
# one is a large projected model sized for a datacenter GPU.
SMALL_1x128 = LstmWorkload("lstm1x128_T100_B1", seed=0, num_layers=1, input_dim=40, hidden=128, proj=0,
                           num_classes=0, batch=1, frames=100, w_range=0.1, output_mode=0)
LSTM_5x500_B1 = LstmWorkload("lstm5x500_C2000_T300_B1", seed=1, num_layers=5, input_dim=40, hidden=500, proj=0,
                             num_classes=2000, batch=1, frames=300, w_range=0.08, forget_bias=1.0)
LSTM_5x500_B256 = LstmWorkload("lstm5x500_C2000_T500_B256", seed=2, num_layers=5, input_dim=40, hidden=500,
                               proj=0, num_classes=2000, batch=256, frames=500, w_range=0.08, forget_bias=1.0,
                               seq_mean_range=0.5)
LSTMP_5x2048P512_B1024 = LstmWorkload("lstmp5x2048p512_C8192_T1000_B1024", seed=4, num_layers=5, input_dim=80,
                                      hidden=2048, proj=512, num_classes=8192, batch=1024, frames=1000,
                                      w_range=0.05)

LSTM_WORKLOADS = {w.name: w for w in (SMALL_1x128, LSTM_5x500_B1, LSTM_5x500_B256, LSTMP_5x2048P512_B1024)}


@dataclass(frozen=True)
class QmatmulShape:
    M: int
    N: int
    K: int


QMATMUL_SEED = 3
QMATMUL_SWEEP = tuple(QmatmulShape(M, KN, KN) for KN in (512, 2048, 8192) for M in (1, 16, 256, 4096, 16384))


def make_qmatmul_operands(shape: QmatmulShape, seed: int = QMATMUL_SEED):
    """fp32 weight W [N, K] ~ N(0, 0.05) and activation A [M, K] = sigmoid of N(0, 2) draws.
    The sigmoid here only shapes the synthetic distribution (values in (0, 1), like gate
    outputs); it is computed in float64 by numpy and is not part of the method under test."""
    rng = np.random.Generator(np.random.PCG64(seed))
    W = rng.normal(0.0, 0.05, (shape.N, shape.K)).astype(np.float32)
    z = rng.normal(0.0, 2.0, (shape.M, shape.K))
    A = (1.0 / (1.0 + np.exp(-z))).astype(np.float32)
    return W, A


def make_matrix(rng: np.random.Generator, rows: int, cols: int, kind: str = "normal") -> np.ndarray:
    if kind == "normal":
        return rng.standard_normal((rows, cols)).astype(np.float32)
    if kind == "uniform":
        return rng.uniform(-1.0, 1.0, (rows, cols)).astype(np.float32)
    raise ValueError(kind)
