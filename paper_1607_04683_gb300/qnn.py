"""Thin Python binding of libqnn (include/qnn.h) with the same call names.

Argument marshalling only: every step of the computation runs in the CUDA library. PyTorch
provides device memory and the current stream. If libqnn.so is missing or cannot be loaded the
calls raise; there is no CPU fallback.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libqnn.so")

QNN_OK = 0
QNN_ERR_INVALID_ARG = 1
QNN_ERR_NONFINITE = 2
QNN_ERR_K_TOO_LARGE = 3
QNN_ERR_CUDA = 4
QNN_ERR_TIMEOUT = 5
QNN_ERR_NO_COOP = 6
QNN_ERR_NO_MEMORY = 7
PER_MATRIX, PER_ROW = 0, 1
OUT_NONE, OUT_QUANT, OUT_FLOAT = 0, 1, 2
K_MAX = 33025

# qnn_qparams {float vmin, vmax, Q; int32 z} as a numpy record (16 bytes)
QPARAMS_DTYPE = np.dtype([("vmin", "<f4"), ("vmax", "<f4"), ("Q", "<f4"), ("z", "<i4")])

# Every symbol the header declares (checked by the CPU test that loads the library).
EXPORTS = ("qnn_status_string", "qnn_device_status", "qnn_quantize", "qnn_qmatmul", "qnn_lstm_param_count",
           "qnn_lstm_model_create", "qnn_lstm_model_destroy", "qnn_lstm_model_weights", "qnn_lstm_forward",
           "qnn_lstm_forward_logits",
           "qnn_profile_enable", "qnn_profile_read", "qnn_measure_peak", "qnn_quantize_matrix_static",
           "qnn_selftest_s64_to_f32", "qnn_stack_frames", "qnn_selftest_wait_timeout", "qnn_selftest_pair_functions", "qnn_lstm_stream_open",
           "qnn_lstm_stream_push", "qnn_lstm_stream_pull", "qnn_lstm_stream_close", "qnn_measure_exchange_floor")


class QnnError(RuntimeError):
    def __init__(self, status: int, where: str = ""):
        self.status = status
        msg = lib().qnn_status_string(status).decode() if _lib is not None else f"status {status}"
        super().__init__(f"{where}: {msg}" if where else msg)


class LstmDesc(C.Structure):
    _fields_ = [("num_layers", C.c_int32), ("input_dim", C.c_int32), ("hidden", C.c_int32),
                ("proj", C.c_int32), ("num_classes", C.c_int32), ("output_mode", C.c_int32),
                ("stack", C.c_int32), ("stack_stride", C.c_int32), ("weight_blocks", C.c_int32)]


_lib = None


def lib():
    """Load libqnn.so (build it first with __graft_entry__.build() or paper_1607_04683_gb300.build)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libqnn.so not built at {LIB_PATH}; run the package build first")
        L = C.CDLL(LIB_PATH)
        P, i64, i32 = C.c_void_p, C.c_int64, C.c_int
        L.qnn_status_string.argtypes = [i32]
        L.qnn_status_string.restype = C.c_char_p
        L.qnn_device_status.argtypes = [P]
        L.qnn_device_status.restype = i32
        L.qnn_quantize.argtypes = [P, i64, i64, i64, i32, P, i64, P, P, P]
        L.qnn_quantize.restype = i32
        L.qnn_qmatmul.argtypes = [P, i64, P, i32, P, i64, i64, P, i64, P, i64, P, i64, P, P, i64, P, P]
        L.qnn_qmatmul.restype = i32
        L.qnn_lstm_param_count.argtypes = [C.POINTER(LstmDesc)]
        L.qnn_lstm_param_count.restype = i64
        L.qnn_lstm_model_create.argtypes = [C.POINTER(LstmDesc), P, C.POINTER(P)]
        L.qnn_lstm_model_create.restype = i32
        L.qnn_lstm_model_destroy.argtypes = [P]
        L.qnn_lstm_model_destroy.restype = None
        L.qnn_lstm_model_weights.argtypes = [P, P, P, C.POINTER(i64)]
        L.qnn_lstm_model_weights.restype = i32
        L.qnn_lstm_forward.argtypes = [P, P, i64, i64, P, P, P, P, P]
        L.qnn_lstm_forward.restype = i32
        L.qnn_lstm_forward_logits.argtypes = [P, P, i64, i64, P, P, P, P, P, P]
        L.qnn_lstm_forward_logits.restype = i32
        L.qnn_profile_enable.argtypes = [i32]
        L.qnn_profile_enable.restype = i32
        L.qnn_profile_read.argtypes = [i32, P, P, P, C.POINTER(i32)]
        L.qnn_profile_read.restype = i32
        L.qnn_measure_peak.argtypes = [i32, C.POINTER(C.c_double)]
        L.qnn_measure_peak.restype = i32
        L.qnn_selftest_s64_to_f32.argtypes = [P, P, i64, P]
        L.qnn_stack_frames.argtypes = [P, i64, i64, i64, i32, i32, P, P]
        L.qnn_selftest_pair_functions.argtypes = [P, i64, P, P]
        L.qnn_selftest_pair_functions.restype = i32
        L.qnn_selftest_wait_timeout.argtypes = [i64, P]
        L.qnn_selftest_wait_timeout.restype = i32
        L.qnn_stack_frames.restype = i32
        L.qnn_selftest_s64_to_f32.restype = i32
        L.qnn_measure_exchange_floor.argtypes = [i32, i32, C.POINTER(C.c_double)]
        L.qnn_measure_exchange_floor.restype = i32
        L.qnn_lstm_stream_open.argtypes = [P, i64, i64, C.c_double, C.POINTER(P)]
        L.qnn_lstm_stream_open.restype = i32
        L.qnn_lstm_stream_push.argtypes = [P, P, i64]
        L.qnn_lstm_stream_push.restype = i32
        L.qnn_lstm_stream_pull.argtypes = [P, P, i64, C.c_double]
        L.qnn_lstm_stream_pull.restype = i32
        L.qnn_lstm_stream_close.argtypes = [P]
        L.qnn_lstm_stream_close.restype = i32
        L.qnn_quantize_matrix_static.argtypes = [P, i64, i64, i64, P, i64, P, P, P, P]
        L.qnn_quantize_matrix_static.restype = i32
        _lib = L
    return _lib


def profile_enable(on: bool = True):
    _check(lib().qnn_profile_enable(1 if on else 0), "qnn_profile_enable")


def measure_peak(kind: int) -> float:
    """Measured peak TOPS of an integer datapath: 0 = mma.sync u8 tensor-core MMA, 1 = dp4a."""
    v = C.c_double(0.0)
    _check(lib().qnn_measure_peak(kind, C.byref(v)), "qnn_measure_peak")
    return v.value


def measure_exchange_floor(cluster_size: int, rounds: int = 20000) -> float:
    """Microseconds per round of the batch-of-few recurrence's per-frame synchronisation skeleton
    (no arithmetic) on one cluster of cluster_size blocks: the floor under a layer's time per frame."""
    v = C.c_double(0.0)
    _check(lib().qnn_measure_exchange_floor(cluster_size, rounds, C.byref(v)), "qnn_measure_exchange_floor")
    return v.value


def selftest_s64_to_f32(values):
    """The device's int64 -> fp32 round-to-nearest conversion of the recovery, on a torch int64
    CUDA tensor; returns a float32 tensor (diagnostic)."""
    import torch
    out = torch.empty(values.shape, dtype=torch.float32, device=values.device)
    _check(lib().qnn_selftest_s64_to_f32(values.data_ptr(), out.data_ptr(), values.numel(),
                                         torch.cuda.current_stream().cuda_stream), "qnn_selftest_s64_to_f32")
    return out


def selftest_pair_functions(values) -> int:
    """Pairs of a float32 CUDA tensor through the gate kernel's paired-instruction functions and
    their one-value forms; returns the number of pairs whose results differ in any bit."""
    import torch
    out = torch.zeros(1, dtype=torch.int64, device=values.device)
    _check(lib().qnn_selftest_pair_functions(values.data_ptr(), values.numel() // 2, out.data_ptr(),
                                             torch.cuda.current_stream().cuda_stream), "qnn_selftest_pair_functions")
    return int(out.item())


def selftest_wait_timeout(limit_ns: int, stream=None):
    """A bounded device wait that nothing ends: raises unless it gave up as designed."""
    _check(lib().qnn_selftest_wait_timeout(int(limit_ns), _stream(stream)), "qnn_selftest_wait_timeout")


def profile_read() -> dict:
    """{kernel name: (launches, total device ms)} since the last read (waits for the events)."""
    cap = 64
    names = (C.c_char_p * cap)()
    ms = (C.c_double * cap)()
    n_l = (C.c_int64 * cap)()
    cnt = C.c_int(0)
    _check(lib().qnn_profile_read(cap, C.cast(names, C.c_void_p), C.cast(ms, C.c_void_p), C.cast(n_l, C.c_void_p),
                                  C.byref(cnt)), "qnn_profile_read")
    return {names[i].decode(): (int(n_l[i]), float(ms[i])) for i in range(min(cnt.value, cap))}


def _check(st: int, where: str):
    if st != QNN_OK:
        raise QnnError(st, where)


def _p(t):
    """Raw pointer of a torch tensor or numpy array (None -> NULL)."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data_as(C.c_void_p)
    return C.c_void_p(t.data_ptr())


def _stream(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream.cuda_stream)


def params_view(p) -> np.ndarray:
    """Device params tensor (int32 [n, 4]) -> numpy records with fields vmin, vmax, Q, z."""
    return p.detach().cpu().numpy().view(QPARAMS_DTYPE).reshape(-1)


def params_tensor(records: np.ndarray, device="cuda"):
    import torch
    raw = np.ascontiguousarray(records, QPARAMS_DTYPE).view(np.int32).reshape(-1, 4)
    return torch.from_numpy(raw.copy()).to(device)


def device_status(stream=None) -> int:
    return int(lib().qnn_device_status(_stream(stream)))


def qnn_quantize(x, granularity=PER_MATRIX, stream=None):
    """x: CUDA fp32 [rows, cols] (row stride may exceed cols). Returns (codes u8, params int32 [n,4],
    code_sums int32 [rows])."""
    import torch
    assert x.is_cuda and x.dtype == torch.float32 and x.dim() == 2 and x.stride(1) == 1
    rows, cols = x.shape
    codes = torch.empty((rows, cols), dtype=torch.uint8, device=x.device)
    params = torch.zeros((1 if granularity == PER_MATRIX else rows, 4), dtype=torch.int32, device=x.device)
    sums = torch.empty(rows, dtype=torch.int32, device=x.device)
    _check(lib().qnn_quantize(_p(x), rows, cols, x.stride(0), granularity, _p(codes), cols, _p(params), _p(sums),
                              _stream(stream)), "qnn_quantize")
    return codes, params, sums


def qnn_qmatmul(A, pa, ga, rsA, W, pw, csW, n_blocks=1, bias=None, want_acc=False, out=None, stream=None):
    """Y = R(A' W'^T) + bias (eq. 1). A u8 [M, K], W u8 [N, K] (CUDA). Returns (Y fp32 [M, N], acc or None)."""
    import torch
    M, K = A.shape
    N, K2 = W.shape
    assert K == K2 and A.stride(1) == 1 and W.stride(1) == 1
    Y = out if out is not None else torch.empty((M, N), dtype=torch.float32, device=A.device)
    acc = torch.empty((M, N), dtype=torch.int32, device=A.device) if want_acc else None
    _check(lib().qnn_qmatmul(_p(A), A.stride(0), _p(pa), ga, _p(rsA), M, K, _p(W), W.stride(0), _p(pw), n_blocks,
                             _p(csW), N, _p(bias), _p(Y), Y.stride(0), _p(acc), _stream(stream)), "qnn_qmatmul")
    return Y, acc


def lstm_desc(num_layers, input_dim, hidden, proj=0, num_classes=0, output_mode=None, stack=0,
              stack_stride=0, weight_blocks=0) -> LstmDesc:
    if output_mode is None:
        output_mode = OUT_QUANT if num_classes > 0 else OUT_NONE
    return LstmDesc(num_layers, input_dim, hidden, proj, num_classes, output_mode, stack, stack_stride,
                    weight_blocks)


def stack_frames(x, n: int, stride: int, out=None, stream=None):
    """Sec. 4 frontend on a CUDA tensor x [B, T, I]: [B, ceil(T/stride), n*I], input t' = frames
    stride*t' .. stride*t' + n - 1 concatenated (the last frame standing in past the end)."""
    import torch
    B, T, I = x.shape
    if out is None:
        out = torch.empty((B, (T + stride - 1) // stride, n * I), dtype=torch.float32, device=x.device)
    _check(lib().qnn_stack_frames(_p(x), B, T, I, n, stride, _p(out), _stream(stream)), "qnn_stack_frames")
    return out


def qnn_lstm_param_count(d: LstmDesc) -> int:
    return int(lib().qnn_lstm_param_count(C.byref(d)))


class LstmModel:
    """Owns a qnn_lstm_model handle: weights quantized offline at construction (Sec. 3.1)."""

    def __init__(self, d: LstmDesc, params):
        self.desc = d
        self.R = d.proj if d.proj > 0 else d.hidden
        n = qnn_lstm_param_count(d)
        if n < 0:
            raise QnnError(QNN_ERR_INVALID_ARG, "qnn_lstm_param_count")
        assert int(params.numel() if hasattr(params, "numel") else params.size) == n
        h = C.c_void_p()
        _check(lib().qnn_lstm_model_create(C.byref(d), _p(params), C.byref(h)), "qnn_lstm_model_create")
        self._h = h

    def close(self):
        if getattr(self, "_h", None) and _lib is not None:
            _lib.qnn_lstm_model_destroy(self._h)
            self._h = None

    __del__ = close

    def weights(self):
        """(codes u8 [param_count] in the packed layout, params records per unit)."""
        n = qnn_lstm_param_count(self.desc)
        codes = np.zeros(n, np.uint8)
        nu = C.c_int64(0)
        _check(lib().qnn_lstm_model_weights(self._h, None, None, C.byref(nu)), "qnn_lstm_model_weights")
        prm = np.zeros(nu.value, QPARAMS_DTYPE)
        _check(lib().qnn_lstm_model_weights(self._h, _p(codes), _p(prm), C.byref(nu)), "qnn_lstm_model_weights")
        return codes, prm

    def forward(self, x, y=None, h_state=None, c_state=None, h_all=None, stream=None, logits=None):
        """x [B, T, I] fp32 (CUDA tensor, or numpy/pinned CPU tensor: copied inside the call).
        Returns y ([B, T, C] or [B, T, R]). A y given in pinned CPU memory receives the posteriors
        from the softmax kernel directly; with any CPU buffer, synchronize the stream before
        reading it. logits: optional [B, T, C] buffer (host or device) that receives the output
        layer's values before the softmax (qnn_lstm_forward_logits)."""
        import torch
        B, T, I = x.shape
        d = self.desc
        ycols = d.num_classes if d.num_classes > 0 else self.R
        if d.stack_stride > 1:  # frame stacking: one network input every stack_stride frames
            T = (T + d.stack_stride - 1) // d.stack_stride
        if y is None:
            if isinstance(x, np.ndarray):
                y = np.empty((B, T, ycols), np.float32)
            else:
                y = torch.empty((B, T, ycols), dtype=torch.float32, device=x.device)
        if logits is None:
            _check(lib().qnn_lstm_forward(self._h, _p(x), B, x.shape[1], _p(y), _p(h_state), _p(c_state),
                                          _p(h_all), _stream(stream)), "qnn_lstm_forward")
        else:
            _check(lib().qnn_lstm_forward_logits(self._h, _p(x), B, x.shape[1], _p(y), _p(logits), _p(h_state),
                                                 _p(c_state), _p(h_all), _stream(stream)), "qnn_lstm_forward_logits")
        return y


class LstmStream:
    """Streaming server mode (qnn_lstm_stream_*): B sequences fed frame by frame to a resident
    kernel; push() appends frames [B, n, I], pull() returns the next frames' outputs [B, n, out]
    (posteriors, or top-layer outputs without an output layer). Host numpy arrays only."""

    def __init__(self, model: LstmModel, B: int, chunk: int = 1024, idle_seconds: float = 10.0):
        self.model, self.B = model, B
        d = model.desc
        self.I = d.input_dim * max(d.stack, 1)
        self.out_dim = d.num_classes if d.num_classes > 0 else model.R
        h = C.c_void_p()
        _check(lib().qnn_lstm_stream_open(model._h, B, chunk, idle_seconds, C.byref(h)), "qnn_lstm_stream_open")
        self._h = h

    def push(self, x: np.ndarray):
        x = np.ascontiguousarray(x, dtype=np.float32)
        assert x.ndim == 3 and x.shape[0] == self.B and x.shape[2] == self.I
        _check(lib().qnn_lstm_stream_push(self._h, _p(x), x.shape[1]), "qnn_lstm_stream_push")

    def pull(self, n: int, timeout: float = 10.0) -> np.ndarray:
        y = np.empty((self.B, n, self.out_dim), np.float32)
        _check(lib().qnn_lstm_stream_pull(self._h, _p(y), n, timeout), "qnn_lstm_stream_pull")
        return y

    def close(self) -> int:
        """Ends the session; returns the first status the kernel recorded (QNN_OK if none)."""
        st = QNN_OK
        if getattr(self, "_h", None) and _lib is not None:
            st = _lib.qnn_lstm_stream_close(self._h)
            self._h = None
        return st

    __del__ = close
