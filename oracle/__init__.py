"""CPU oracle for 8-bit quantized LSTM inference (Alvarez et al., INTERSPEECH 2016).

TEST INFRASTRUCTURE ONLY: the test suite, the smoke check and the benchmark's CPU-baseline leg
are the only users. The product path never imports this package; it shares no code with the CUDA
library. The arithmetic lives in ``qnn_oracle.c`` (plain C, fp32 op by op as the paper's
Sec. 3 and 3.1 define it, integer products exact); this module compiles it with gcc and marshals
numpy arrays through ctypes.

Functions and the passages they follow:
  params_from_range  Sec. 3 "Quantizing" (S = 255, Q = S/R) and eq. (2) (offset round(Q Vmin))
  quantize           Sec. 3 "Quantizing", eq. (2); per matrix or per row (Sec. 3.1 granularity)
  recover            eq. (3)
  qmatmul            eq. (1): integer product of offset-applied codes, recovered by 1/(Qa Qb)
  exp_, sigmoid, tanh  pinned fp32 transcendentals used by both sides
  lstm_forward       Sec. 3.1 / Fig. 1 layer scheme applied to an LSTM(P) stack and output layer
  lstm_quantize_weights  offline weight quantization, one unit per gate matrix (Sec. 3.1)

Parity pins for every function are in tests/test_oracle_pins.py; end-to-end LSTM outputs are
"parity unpinned" against the paper's own numbers (its only numbers are word error rates on
proprietary data), and pinned instead by the reductions and invariants those tests check.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "qnn_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]

OK, ERR_INVALID_ARG, ERR_NONFINITE, ERR_K_TOO_LARGE = 0, 1, 2, 3
PER_MATRIX, PER_ROW = 0, 1
OUT_NONE, OUT_QUANT, OUT_FLOAT = 0, 1, 2
K_MAX = 33025

_lock = threading.Lock()
_lib = None


class QParams(C.Structure):
    _fields_ = [("vmin", C.c_float), ("vmax", C.c_float), ("Q", C.c_float), ("z", C.c_int32)]


QPARAMS_DTYPE = np.dtype([("vmin", "<f4"), ("vmax", "<f4"), ("Q", "<f4"), ("z", "<i4")])


class LstmDesc(C.Structure):
    _fields_ = [("num_layers", C.c_int32), ("input_dim", C.c_int32), ("hidden", C.c_int32),
                ("proj", C.c_int32), ("num_classes", C.c_int32), ("output_mode", C.c_int32),
                ("weight_blocks", C.c_int32)]


def build(force: bool = False) -> str:
    """Compile liboracle.so next to its source (gcc, no GPU needed)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", *CFLAGS, "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            P = C.c_void_p
            i64 = C.c_int64
            L.orc_params_from_range.argtypes = [C.c_float, C.c_float, C.POINTER(QParams)]
            L.orc_params_from_range.restype = None
            L.orc_quantize.argtypes = [P, i64, i64, i64, C.c_int, P, i64, P, P]
            L.orc_quantize.restype = C.c_int
            L.orc_recover.argtypes = [C.c_uint8, C.POINTER(QParams)]
            L.orc_recover.restype = C.c_float
            L.orc_code.argtypes = [C.c_float, C.POINTER(QParams)]
            L.orc_code.restype = C.c_uint8
            L.orc_qmatmul.argtypes = [P, i64, P, C.c_int, i64, i64, P, i64, P, i64, i64, P, P, i64, P, P]
            L.orc_qmatmul.restype = C.c_int
            for name in ("orc_exp", "orc_sigmoid", "orc_tanh"):
                getattr(L, name).argtypes = [C.c_float]
                getattr(L, name).restype = C.c_float
            L.orc_lstm_param_count.argtypes = [C.POINTER(LstmDesc)]
            L.orc_lstm_param_count.restype = i64
            L.orc_lstm_forward.argtypes = [C.POINTER(LstmDesc), P, P, i64, i64, P, P, P, P, P]
            L.orc_lstm_forward.restype = C.c_int
            L.orc_lstm_quantize_weights.argtypes = [C.POINTER(LstmDesc), P, P, P, C.POINTER(i64)]
            L.orc_stack_frames.argtypes = [P, i64, i64, i64, C.c_int, C.c_int, P]
            L.orc_stack_frames.restype = C.c_int
            L.orc_lstm_quantize_weights.restype = C.c_int
            _lib = L
    return _lib


class OracleError(RuntimeError):
    def __init__(self, status: int):
        super().__init__(f"oracle status {status}")
        self.status = status


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _check(st):
    if st != OK:
        raise OracleError(st)


def params_from_range(vmin: float, vmax: float) -> dict:
    p = QParams()
    lib().orc_params_from_range(C.c_float(vmin), C.c_float(vmax), C.byref(p))
    return {"vmin": p.vmin, "vmax": p.vmax, "Q": p.Q, "z": p.z}


def _as_qparams(d) -> QParams:
    return QParams(d["vmin"], d["vmax"], d["Q"], int(d["z"]))


def quantize(x: np.ndarray, granularity: int = PER_MATRIX):
    """fp32 [rows, cols] -> (codes u8 [rows, cols], params structured [1 or rows], row sums i32)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    if x.ndim == 1:
        x = x[None, :]
    rows, cols = x.shape
    codes = np.empty((rows, cols), np.uint8)
    params = np.zeros(1 if granularity == PER_MATRIX else rows, QPARAMS_DTYPE)
    sums = np.empty(rows, np.int32)
    _check(lib().orc_quantize(_ptr(x), rows, cols, cols, granularity, _ptr(codes), cols, _ptr(params), _ptr(sums)))
    return codes, params, sums


def code(v: float, p: dict) -> int:
    return int(lib().orc_code(C.c_float(v), C.byref(_as_qparams(p))))


def recover(codes: np.ndarray, p) -> np.ndarray:
    """Eq. (3) elementwise, codes with one parameter set (dict or structured scalar)."""
    q = _as_qparams(p)
    f = lib().orc_recover
    flat = np.asarray(codes, np.uint8).ravel()
    return np.array([f(int(c), C.byref(q)) for c in flat], np.float32).reshape(np.shape(codes))


def qmatmul(A, pa, ga, W, pw, n_blocks=1, bias=None, want=("y", "acc", "S")):
    """Eq. (1). A u8 [M, K] with params pa (1 or M), W u8 [N, K] with n_blocks params.
    Returns dict with y (fp32 [M, N]), acc (int32 raw code product), S (int64 offset product)."""
    A = np.ascontiguousarray(A, np.uint8)
    W = np.ascontiguousarray(W, np.uint8)
    M, K = A.shape
    N, K2 = W.shape
    assert K == K2
    pa = np.ascontiguousarray(pa, QPARAMS_DTYPE)
    pw = np.ascontiguousarray(pw, QPARAMS_DTYPE)
    out = {}
    y = np.empty((M, N), np.float32) if "y" in want else None
    acc = np.empty((M, N), np.int32) if "acc" in want else None
    S = np.empty((M, N), np.int64) if "S" in want else None
    b = None if bias is None else np.ascontiguousarray(bias, np.float32)
    _check(lib().orc_qmatmul(_ptr(A), K, _ptr(pa), ga, M, K, _ptr(W), K, _ptr(pw), n_blocks, N, _ptr(b),
                             _ptr(y), N, _ptr(acc), _ptr(S)))
    if y is not None:
        out["y"] = y
    if acc is not None:
        out["acc"] = acc
    if S is not None:
        out["S"] = S
    return out


def exp_(x: float) -> float:
    return float(lib().orc_exp(C.c_float(x)))


def sigmoid(x: float) -> float:
    return float(lib().orc_sigmoid(C.c_float(x)))


def tanh(x: float) -> float:
    return float(lib().orc_tanh(C.c_float(x)))


def desc(num_layers, input_dim, hidden, proj=0, num_classes=0, output_mode=None, weight_blocks=0) -> LstmDesc:
    """weight_blocks: quantization units per weight matrix, as equal blocks of rows (Sec. 3.1)."""
    if output_mode is None:
        output_mode = OUT_QUANT if num_classes > 0 else OUT_NONE
    return LstmDesc(num_layers, input_dim, hidden, proj, num_classes, output_mode, weight_blocks)


def lstm_param_count(d: LstmDesc) -> int:
    return int(lib().orc_lstm_param_count(C.byref(d)))


def lstm_forward(d: LstmDesc, params: np.ndarray, x: np.ndarray, h0=None, c0=None, want_h_all=False,
                 want_logits=False):
    """x fp32 [B, T, I] -> dict(y, h, c[, h_all][, logits]). h0/c0: [L, B, R] / [L, B, H] or None."""
    params = np.ascontiguousarray(params, np.float32)
    assert params.size == lstm_param_count(d)
    x = np.ascontiguousarray(x, np.float32)
    B, T, I = x.shape
    assert I == d.input_dim
    L, H = d.num_layers, d.hidden
    R = d.proj if d.proj > 0 else H
    Cn = d.num_classes
    y = np.empty((B, T, Cn if Cn > 0 else R), np.float32)
    h = np.zeros((L, B, R), np.float32) if h0 is None else np.array(h0, np.float32, copy=True)
    c = np.zeros((L, B, H), np.float32) if c0 is None else np.array(c0, np.float32, copy=True)
    h_all = np.empty((L, B, T, R), np.float32) if want_h_all else None
    logits = np.empty((B, T, Cn), np.float32) if (want_logits and Cn > 0) else None
    _check(lib().orc_lstm_forward(C.byref(d), _ptr(params), _ptr(x), B, T, _ptr(y), _ptr(h), _ptr(c),
                                  _ptr(h_all), _ptr(logits)))
    out = {"y": y, "h": h, "c": c}
    if h_all is not None:
        out["h_all"] = h_all
    if logits is not None:
        out["logits"] = logits
    return out


def lstm_quantize_weights(d: LstmDesc, params: np.ndarray):
    """Offline weight codes in packed order (u8) and one params entry per unit."""
    params = np.ascontiguousarray(params, np.float32)
    n = lstm_param_count(d)
    codes = np.zeros(n, np.uint8)
    nb = max(1, d.weight_blocks)
    qp = np.zeros(nb * (9 * d.num_layers + 1), QPARAMS_DTYPE)
    nu = C.c_int64(0)
    _check(lib().orc_lstm_quantize_weights(C.byref(d), _ptr(params), _ptr(codes), _ptr(qp), C.byref(nu)))
    return codes, qp[: nu.value]


def stack_frames(x: np.ndarray, n: int, stride: int) -> np.ndarray:
    """Sec. 4 frontend (reading R9): x [B, T, I] -> [B, ceil(T/stride), n*I]; input t' concatenates
    frames stride*t' .. stride*t' + n - 1, the last frame standing in past the end."""
    x = np.ascontiguousarray(x, np.float32)
    B, T, I = x.shape
    out = np.empty((B, (T + stride - 1) // stride, n * I), np.float32)
    _check(lib().orc_stack_frames(_ptr(x), B, T, I, n, stride, _ptr(out)))
    return out
