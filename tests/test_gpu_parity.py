"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the same seeded inputs.

Bar: codes, parameters, code sums and int32 accumulators bit-exact; every LSTM layer output
bit-exact (the whole recurrence is the same sequence of fp32 operations on both sides, so any
difference would be a bug); the 8-bit output layer's logits bit-exact; posteriors within 1e-4
absolute and 1e-5 relative (their sums run in a different order on the GPU). The rules are in
tests/parity.py.
"""
import ctypes
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import oracle
import parity
from paper_1607_04683_gb300 import inputs

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
    assert q.device_status() == q.QNN_OK
    return q


def gpu(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


# ------------------------------------------------------------------------------------------
# qnn_quantize
# ------------------------------------------------------------------------------------------

QUANT_SHAPES = [(1, 1), (1, 3), (3, 5), (7, 40), (9, 128), (33, 500), (300, 40), (17, 1000), (5, 8192), (1025, 77)]


@pytest.mark.parametrize("rows,cols", QUANT_SHAPES)
@pytest.mark.parametrize("gran", [0, 1])
def test_quantize_bit_exact(qnn, rows, cols, gran):
    r = rng(rows * 1000 + cols)
    x = (r.normal(0.3, 1.7, (rows, cols)) * r.uniform(0.01, 10, (rows, 1))).astype(np.float32)
    codes, params, sums = qnn.qnn_quantize(gpu(x), gran)
    assert qnn.device_status() == qnn.QNN_OK
    c_ref, p_ref, s_ref = oracle.quantize(x, gran)
    assert np.array_equal(codes.cpu().numpy(), c_ref)
    assert np.array_equal(sums.cpu().numpy(), s_ref)
    p = qnn.params_view(params)
    for f in ("vmin", "vmax", "Q", "z"):
        assert np.array_equal(p[f], p_ref[f]), f


def test_quantize_strided_and_degenerate_rows(qnn):
    r = rng(5)
    big = r.normal(0, 1, (64, 203)).astype(np.float32)
    big[3] = 0.0
    big[7] = -2.5
    big[11, :] = 1e-3
    big[11, 5] = np.nextafter(np.float32(1e-3), np.float32(1))
    view = gpu(big)[:, 3:190]  # row stride 203, unaligned start
    codes, params, sums = qnn.qnn_quantize(view, qnn.PER_ROW)
    c_ref, p_ref, s_ref = oracle.quantize(np.ascontiguousarray(big[:, 3:190]), oracle.PER_ROW)
    assert np.array_equal(codes.cpu().numpy(), c_ref)
    assert np.array_equal(sums.cpu().numpy(), s_ref)
    p = qnn.params_view(params)
    for f in ("vmin", "vmax", "Q", "z"):
        assert np.array_equal(p[f], p_ref[f]), f


@pytest.mark.parametrize("cols,ld", [(190, 256), (1022, 1024), (1024, 1028), (1025, 1028), (509, 512), (2, 4)])
def test_quantize_per_row_aligned_ragged(qnn, cols, ld):
    # 16-byte aligned rows whose length is not a multiple of 4 (ragged last float4), at and past
    # the 1024-value register-resident limit
    r = rng(cols * 7 + ld)
    big = (r.normal(-0.2, 2.0, (37, ld)) * r.uniform(0.1, 5, (37, 1))).astype(np.float32)
    codes, params, sums = qnn.qnn_quantize(gpu(big)[:, :cols], qnn.PER_ROW)
    assert qnn.device_status() == qnn.QNN_OK
    c_ref, p_ref, s_ref = oracle.quantize(np.ascontiguousarray(big[:, :cols]), oracle.PER_ROW)
    assert np.array_equal(codes.cpu().numpy(), c_ref)
    assert np.array_equal(sums.cpu().numpy(), s_ref)
    p = qnn.params_view(params)
    for f in ("vmin", "vmax", "Q", "z"):
        assert np.array_equal(p[f], p_ref[f]), f


def test_quantize_large_matrix_per_matrix(qnn):
    # config-4 size activation: 16384 x 8192, per-matrix unit; codes checked on sampled rows.
    shape = inputs.QmatmulShape(16384, 8192, 8192)
    W, A = inputs.make_qmatmul_operands(shape)
    Ag = gpu(A)
    codes, params, sums = qnn.qnn_quantize(Ag, qnn.PER_MATRIX)
    p = qnn.params_view(params)[0]
    assert p["vmin"] == A.min() and p["vmax"] == A.max()
    ref = oracle.params_from_range(float(A.min()), float(A.max()))
    assert p["Q"] == np.float32(ref["Q"]) and p["z"] == ref["z"]
    rows = rng(1).choice(shape.M, 64, replace=False)
    cs = codes[torch.from_numpy(rows).cuda()].cpu().numpy()
    for i, row in enumerate(rows):
        exp = np.array([oracle.code(float(v), ref) for v in A[row, ::97]], np.uint8)
        assert np.array_equal(cs[i, ::97], exp)
        assert sums[int(row)].item() == int(cs[i].astype(np.int64).sum())


def test_quantize_nonfinite_reported(qnn):
    x = np.ones((4, 33), np.float32)
    x[2, 7] = np.nan
    qnn.qnn_quantize(gpu(x), qnn.PER_ROW)
    assert qnn.device_status() == qnn.QNN_ERR_NONFINITE
    assert qnn.device_status() == qnn.QNN_OK  # cleared by the read
    x[2, 7] = np.inf
    qnn.qnn_quantize(gpu(x), qnn.PER_MATRIX)
    assert qnn.device_status() == qnn.QNN_ERR_NONFINITE


def test_quantize_rejects_host_pointers(qnn):
    import ctypes as C
    x = np.ones((2, 8), np.float32)
    codes = np.zeros((2, 8), np.uint8)
    prm = np.zeros(2, qnn.QPARAMS_DTYPE)
    st = qnn.lib().qnn_quantize(x.ctypes.data_as(C.c_void_p), 2, 8, 8, 1, codes.ctypes.data_as(C.c_void_p), 8,
                                prm.ctypes.data_as(C.c_void_p), None, None)
    assert st == qnn.QNN_ERR_INVALID_ARG


# ------------------------------------------------------------------------------------------
# qnn_qmatmul
# ------------------------------------------------------------------------------------------

def _operands(M, N, K, ga, seed, n_blocks=1):
    r = rng(seed)
    A = r.normal(0.2, 1.0, (M, K)).astype(np.float32)
    Wf = [r.uniform(-s, s, (N // n_blocks, K)).astype(np.float32) for s in np.linspace(0.05, 0.5, n_blocks)]
    ca, pa, ra = oracle.quantize(A, ga)
    parts = [oracle.quantize(w, oracle.PER_MATRIX) for w in Wf]
    cw = np.concatenate([p[0] for p in parts])
    pw = np.concatenate([p[1] for p in parts])
    cs = np.concatenate([p[2] for p in parts])
    bias = r.normal(0, 1, N).astype(np.float32)
    return ca, pa, ra, cw, pw, cs, bias


MM_SHAPES = [(1, 8, 1), (1, 4, 40), (3, 5, 7), (16, 64, 64), (130, 130, 100), (257, 260, 500), (300, 2000, 40),
             (64, 96, 1000), (200, 136, 2048)]


@pytest.mark.parametrize("M,N,K", MM_SHAPES)
@pytest.mark.parametrize("ga", [0, 1])
def test_qmatmul_bit_exact(qnn, M, N, K, ga):
    nb = 4 if N % 4 == 0 else 1
    ca, pa, ra, cw, pw, cs, bias = _operands(M, N, K, ga, M * 7 + N * 3 + K, nb)
    Y, acc = qnn.qnn_qmatmul(gpu(ca), qnn.params_tensor(pa), ga, gpu(ra), gpu(cw), qnn.params_tensor(pw), gpu(cs),
                             n_blocks=nb, bias=gpu(bias), want_acc=True)
    ref = oracle.qmatmul(ca, pa, ga, cw, pw, n_blocks=nb, bias=bias)
    assert np.array_equal(acc.cpu().numpy(), ref["acc"])
    assert np.array_equal(Y.cpu().numpy(), ref["y"])


def test_qmatmul_unaligned_leading_dims(qnn):
    M, N, K = 37, 45, 99
    ca, pa, ra, cw, pw, cs, _ = _operands(M, N, K, 1, 11)
    Abig = np.zeros((M, K + 5), np.uint8)
    Abig[:, 2:2 + K] = ca
    Ag = gpu(Abig)[:, 2:2 + K]
    Y, acc = qnn.qnn_qmatmul(Ag, qnn.params_tensor(pa), 1, gpu(ra), gpu(cw), qnn.params_tensor(pw), gpu(cs),
                             want_acc=True)
    ref = oracle.qmatmul(ca, pa, 1, cw, pw)
    assert np.array_equal(acc.cpu().numpy(), ref["acc"]) and np.array_equal(Y.cpu().numpy(), ref["y"])


def test_qmatmul_k_max_all_255(qnn):
    K = oracle.K_MAX
    a = np.full((2, K), 255, np.uint8)
    p = np.zeros(1, qnn.QPARAMS_DTYPE)
    p[0] = (0.0, 1.0, 255.0, 0)
    rs = np.full(2, 255 * K, np.int32)
    Y, acc = qnn.qnn_qmatmul(gpu(a), qnn.params_tensor(p), 0, gpu(rs), gpu(a), qnn.params_tensor(p), gpu(rs),
                             want_acc=True)
    assert int(acc[0, 0].item()) == K * 65025 == 2147450625
    with pytest.raises(qnn.QnnError) as e:
        b = np.full((1, K + 1), 1, np.uint8)
        qnn.qnn_qmatmul(gpu(b), qnn.params_tensor(p), 0, gpu(rs[:1]), gpu(b), qnn.params_tensor(p), gpu(rs[:1]))
    assert e.value.status == qnn.QNN_ERR_K_TOO_LARGE


@pytest.mark.parametrize("KN", [512, 2048, 8192])
def test_qmatmul_sweep_full_size_sampled(qnn, KN):
    # The standalone sweep's largest M at each K = N, fp32 in: quantize both operands on the GPU
    # (per matrix), product; compared on a sample of rows and columns the oracle computes.
    shape = inputs.QmatmulShape(16384, KN, KN)
    W, A = inputs.make_qmatmul_operands(shape)
    ca, pa, ra = qnn.qnn_quantize(gpu(A), qnn.PER_MATRIX)
    cw, pw, cs = qnn.qnn_quantize(gpu(W), qnn.PER_MATRIX)
    Y, acc = qnn.qnn_qmatmul(ca, pa, 0, ra, cw, pw, cs, want_acc=True)
    r = rng(KN)
    rows = np.sort(r.choice(shape.M, 48, replace=False))
    cols = np.sort(r.choice(shape.N, 48, replace=False))
    c_a, p_a, _ = oracle.quantize(A, oracle.PER_MATRIX)
    c_w, p_w, _ = oracle.quantize(W, oracle.PER_MATRIX)
    assert np.array_equal(qnn.params_view(pa), p_a) and np.array_equal(qnn.params_view(pw), p_w)
    ref = oracle.qmatmul(c_a[rows], p_a, 0, c_w[cols], p_w)
    ri, ci = torch.from_numpy(rows).cuda(), torch.from_numpy(cols).cuda()
    assert np.array_equal(acc[ri][:, ci].cpu().numpy(), ref["acc"])
    assert np.array_equal(Y[ri][:, ci].cpu().numpy(), ref["y"])


# ------------------------------------------------------------------------------------------
# qnn_lstm_forward
# ------------------------------------------------------------------------------------------

def _small(name="t", L=2, I=7, H=9, P=0, C=0, B=2, T=6, seed=5, mode=None, fb=1.0, w=0.5, mu=0.0, wo=0.0):
    return inputs.LstmWorkload(name, seed=seed, num_layers=L, input_dim=I, hidden=H, proj=P, num_classes=C,
                               batch=B, frames=T, w_range=w, forget_bias=fb, seq_mean_range=mu,
                               output_mode=(mode if mode is not None else (1 if C > 0 else 0)), out_w_range=wo)


def _gpu_forward(qnn, wl, params, x, h_all=True, h0=None, c0=None, logits=True):
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    model = qnn.LstmModel(d, gpu(params))
    B, T, _ = x.shape
    ha = torch.empty((wl.num_layers, B, T, wl.R), dtype=torch.float32, device="cuda") if h_all else None
    hs = gpu(h0) if h0 is not None else torch.zeros((wl.num_layers, B, wl.R), dtype=torch.float32, device="cuda")
    cs = gpu(c0) if c0 is not None else torch.zeros((wl.num_layers, B, wl.hidden), dtype=torch.float32, device="cuda")
    lg = None
    if logits and wl.num_classes > 0:
        lg = torch.full((B, T, wl.num_classes), float("nan"), dtype=torch.float32, device="cuda")
    y = model.forward(gpu(x), h_state=hs, c_state=cs, h_all=ha, logits=lg)
    assert qnn.device_status() == qnn.QNN_OK
    out = {"y": y.cpu().numpy(), "h": hs.cpu().numpy(), "c": cs.cpu().numpy(), "model": model}
    if h_all:
        out["h_all"] = ha.cpu().numpy()
    if lg is not None:
        out["logits"] = lg.cpu().numpy()
    return out


def _compare(got, ref, wl, params=None):
    w_out = wl.out_weights(params) if (params is not None and wl.num_classes > 0) else None
    parity.compare(got, ref, wl.num_layers, wl.num_classes, wl.output_mode, w_out)


def _oracle(wl, params, x, **kw):
    d = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    kw.setdefault("want_logits", wl.num_classes > 0)
    return oracle.lstm_forward(d, params, x, **kw)


SMALL_CASES = [dict(), dict(L=1, I=3, H=4, B=1, T=9), dict(L=3, H=16, C=11, B=3), dict(L=2, H=33, I=40, C=5, B=17, T=4),
               dict(L=2, I=6, H=10, P=4, C=7, B=2, T=5), dict(L=2, I=80, H=130, P=48, C=70, B=20, T=6),
               dict(L=2, H=12, C=5, mode=2), dict(L=1, I=40, H=500, B=70, T=3, C=2000, w=0.08),
               dict(L=2, I=40, H=64, C=9, B=6, T=5), dict(L=2, I=40, H=50, P=16, C=9, B=6, T=4),
               dict(L=3, I=5, H=8, B=65, T=3, mu=0.5),
               # output weights wide enough that the posteriors are far from uniform (logits over
               # several units), on the batch-of-few, integer-MMA and tensor-core paths
               dict(L=2, I=40, H=64, C=2000, B=2, T=7, w=0.3, wo=1.0),
               dict(L=2, I=40, H=64, C=2000, B=9, T=4, w=0.3, wo=1.0),
               dict(L=2, I=40, H=64, P=32, C=2000, B=70, T=3, w=0.3, wo=2.0),
               dict(L=2, I=40, H=64, C=300, B=9, T=4, w=0.3, wo=1.0, mode=2)]


@pytest.mark.parametrize("cfg", SMALL_CASES)
def test_lstm_small_bit_exact(qnn, cfg):
    wl = _small(**cfg)
    params, x = wl.make()
    got = _gpu_forward(qnn, wl, params, x)
    ref = _oracle(wl, params, x, want_h_all=True)
    _compare(got, ref, wl, params)
    if wl.out_w_range > 0:  # the case is meant to spread the posteriors: check that it does
        assert ref["y"].max() > 5.0 / wl.num_classes and ref["y"].min() < 0.1 / wl.num_classes


def test_lstm_weight_codes_bit_exact(qnn):
    wl = _small(L=2, I=40, H=37, P=12, C=9)
    params, _ = wl.make()
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes)
    model = qnn.LstmModel(d, gpu(params))
    codes, prm = model.weights()
    c_ref, p_ref = oracle.lstm_quantize_weights(oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj,
                                                            wl.num_classes), params)
    assert np.array_equal(codes, c_ref)
    assert np.array_equal(prm.view(np.int32), p_ref.view(np.int32))


def test_lstm_streaming_state_and_host_buffers(qnn):
    wl = _small(L=3, H=20, C=6, B=4, T=12)
    params, x = wl.make()
    full = _gpu_forward(qnn, wl, params, x)
    a = _gpu_forward(qnn, wl, params, x[:, :5])
    b = _gpu_forward(qnn, wl, params, x[:, 5:], h0=a["h"], c0=a["c"])
    assert np.array_equal(np.concatenate([a["h_all"], b["h_all"]], 2), full["h_all"])
    assert np.array_equal(b["h"], full["h"]) and np.array_equal(b["c"], full["c"])
    # host (numpy) buffers through the same call
    y_host = full["model"].forward(x)
    assert np.array_equal(y_host, full["y"])


@pytest.mark.parametrize("path,B,mode", [("small", 2, 1), ("small", 4, 1), ("tc", 64, 1), ("layerwise", 5, 1),
                                         ("layerwise", 5, 2)])
def test_lstm_posteriors_into_pinned_host_memory(qnn, path, B, mode, monkeypatch):
    # a y in pinned host memory is written by the softmax kernel itself (no staging copy): the
    # same posteriors as a device y, bit for bit, with pinned or pageable inputs; a pageable y
    # takes the copy
    monkeypatch.setenv("QNN_LSTM_PATH", path)
    wl = _small(L=2, I=8, H=32, C=300, B=B, T=5, mode=mode)
    params, x = wl.make()
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    model = qnn.LstmModel(d, gpu(params))
    y_dev = model.forward(gpu(x))
    torch.cuda.synchronize()
    y_dev = y_dev.cpu().numpy()
    parity.check_posteriors(y_dev, _oracle(wl, params, x)["y"])
    for xin in (torch.from_numpy(x).pin_memory(), x):
        y_pin = torch.full((B, wl.frames, wl.num_classes), float("nan")).pin_memory()
        model.forward(xin, y=y_pin)
        torch.cuda.synchronize()
        assert np.array_equal(y_pin.numpy(), y_dev)
    y_np = model.forward(x)
    torch.cuda.synchronize()
    assert np.array_equal(y_np, y_dev)
    assert qnn.device_status() == qnn.QNN_OK


@pytest.mark.parametrize("path,B", [("small", 2), ("layerwise", 5), ("tc", 64)])
def test_lstm_logits_into_host_memory(qnn, path, B, monkeypatch):
    # qnn_lstm_forward_logits with the logits in pinned and in pageable host memory: the same bits
    # as into device memory and as the oracle's
    monkeypatch.setenv("QNN_LSTM_PATH", path)
    wl = _small(L=2, I=8, H=32, C=300, B=B, T=5, wo=1.0)
    params, x = wl.make()
    ref = _oracle(wl, params, x)
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    model = qnn.LstmModel(d, gpu(params))
    for lg in (torch.full((B, wl.frames, wl.num_classes), float("nan")).pin_memory(),
               np.full((B, wl.frames, wl.num_classes), np.nan, np.float32)):
        y = model.forward(gpu(x), logits=lg)
        torch.cuda.synchronize()
        lgn = lg.numpy() if hasattr(lg, "numpy") else lg
        parity.check_logits(lgn, ref["logits"], 1)
        parity.check_posteriors(y.cpu().numpy(), ref["y"])
    assert qnn.device_status() == qnn.QNN_OK


def test_lstm_logits_need_an_output_layer(qnn):
    wl = _small(L=1, H=8, B=1, T=3)
    params, x = wl.make()
    model = qnn.LstmModel(qnn.lstm_desc(1, wl.input_dim, wl.hidden), gpu(params))
    lg = torch.empty((1, 3, 4), dtype=torch.float32, device="cuda")
    with pytest.raises(qnn.QnnError) as e:
        model.forward(gpu(x), logits=lg)
    assert e.value.status == qnn.QNN_ERR_INVALID_ARG


def test_lstm_nonfinite_input_reported(qnn):
    wl = _small(L=1, H=8, B=1, T=3)
    params, x = wl.make()
    x[0, 1, 2] = np.nan
    d = qnn.lstm_desc(1, wl.input_dim, wl.hidden)
    model = qnn.LstmModel(d, gpu(params))
    model.forward(gpu(x))
    assert qnn.device_status() == qnn.QNN_ERR_NONFINITE


def test_config_small_1x128_full(qnn):
    wl = inputs.SMALL_1x128
    params, x = wl.make()
    got = _gpu_forward(qnn, wl, params, x)
    ref = _oracle(wl, params, x, want_h_all=True)
    _compare(got, ref, wl, params)


def test_config_5x500_b1_full(qnn):
    # the batch-1 workload, whole: 5 x 500 cells, 2000 classes, T = 300
    wl = inputs.LSTM_5x500_B1
    params, x = wl.make()
    got = _gpu_forward(qnn, wl, params, x)
    ref = _oracle(wl, params, x, want_h_all=True)
    _compare(got, ref, wl, params)


def _sequences_by_oracle(wl, params, x, seqs):
    """The oracle on single sequences, in threads (its C calls release the interpreter lock);
    per-row quantization makes every sequence independent of its batch-mates."""
    with ThreadPoolExecutor(max_workers=len(seqs)) as ex:
        return list(ex.map(lambda b: _oracle(wl, params, x[b:b + 1]), seqs))


def _check_sequence(got, ref, b, frames=slice(None)):
    assert np.array_equal(got["h"][:, b], ref["h"][:, 0]) and np.array_equal(got["c"][:, b], ref["c"][:, 0])
    parity.check_logits(got["logits"][b, frames], ref["logits"][0, frames], 1)
    parity.check_posteriors(got["y"][b, frames], ref["y"][0, frames])


def test_config_5x500_b256_sampled(qnn):
    # batch 256 x 500 frames on the GPU; the oracle recomputes two whole sequences: final state,
    # logits (bit-exact) and posteriors of every frame
    wl = inputs.LSTM_5x500_B256
    params, x = wl.make()
    got = _gpu_forward(qnn, wl, params, x, h_all=False)
    seqs = (0, 173)
    for b, ref in zip(seqs, _sequences_by_oracle(wl, params, x, seqs)):
        _check_sequence(got, ref, b)


def test_config_lstmp_2048_b1024_full_length(qnn):
    # the large projected model at its full size (batch 1024, T = 1000: the recurrence through all
    # 1000 steps of the tensor-core path); the oracle recomputes two whole sequences, about a
    # minute each: final (h, c) of every layer bit-exact, logits bit-exact and posteriors on every
    # 7th frame
    wl = inputs.LSTMP_5x2048P512_B1024
    params, x = wl.make()
    B, T = wl.batch, wl.frames
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    model = qnn.LstmModel(d, gpu(params))
    hs = torch.zeros((wl.num_layers, B, wl.R), dtype=torch.float32, device="cuda")
    cs = torch.zeros((wl.num_layers, B, wl.hidden), dtype=torch.float32, device="cuda")
    lg = torch.empty((B, T, wl.num_classes), dtype=torch.float32, device="cuda")
    y = model.forward(gpu(x), h_state=hs, c_state=cs, logits=lg)
    torch.cuda.synchronize()
    assert qnn.device_status() == qnn.QNN_OK
    seqs = (611, 5)
    frames = slice(0, T, 7)
    got = {"h": hs.cpu().numpy(), "c": cs.cpu().numpy()}
    got["logits"] = {b: lg[b, frames].cpu().numpy() for b in seqs}
    got["y"] = {b: y[b, frames].cpu().numpy() for b in seqs}
    del y, lg
    model.close()
    torch.cuda.empty_cache()
    for b, ref in zip(seqs, _sequences_by_oracle(wl, params, x, seqs)):
        assert np.array_equal(got["h"][:, b], ref["h"][:, 0]) and np.array_equal(got["c"][:, b], ref["c"][:, 0])
        parity.check_logits(got["logits"][b], ref["logits"][0, frames], 1)
        parity.check_posteriors(got["y"][b], ref["y"][0, frames])


# ------------------------------------------------------------------------------------------
# The two forward paths: batch-of-few cluster pipeline and layer-by-layer
# ------------------------------------------------------------------------------------------

PATH_CASES = [dict(L=1, I=40, H=128, B=1, T=20), dict(L=3, I=40, H=100, C=37, B=2, T=9),
              dict(L=2, I=13, H=500, C=2000, B=4, T=5, w=0.08), dict(L=5, I=40, H=33, C=3, B=3, T=4)]


@pytest.mark.parametrize("cfg", PATH_CASES)
def test_small_and_layerwise_paths_agree(qnn, cfg, monkeypatch):
    wl = _small(**cfg)
    params, x = wl.make()
    ref = _oracle(wl, params, x, want_h_all=True)
    outs = {}
    for path in ("small", "layerwise"):
        monkeypatch.setenv("QNN_LSTM_PATH", path)
        qnn.profile_read()
        qnn.profile_enable(True)
        got = _gpu_forward(qnn, wl, params, x)
        qnn.profile_enable(False)
        kernels = qnn.profile_read()
        assert ("lstm_small" in kernels) == (path == "small"), kernels
        _compare(got, ref, wl, params)
        outs[path] = got
    assert np.array_equal(outs["small"]["y"], outs["layerwise"]["y"])


# Tensor-core recurrence (large batches): forced on small cases, every tile width
TC_CASES = [dict(L=1, I=40, H=128, B=5, T=6), dict(L=2, I=40, H=100, C=37, B=130, T=4),
            dict(L=2, I=24, H=256, P=96, C=11, B=33, T=5), dict(L=1, I=40, H=500, B=256, T=3, w=0.08, mu=0.5),
            dict(L=1, I=8, H=1024, B=64, T=2, w=0.05), dict(L=2, I=80, H=1100, P=64, C=20, B=40, T=3, w=0.05),
            dict(L=3, I=5, H=8, B=3, T=4, mu=0.5), dict(L=1, I=40, H=800, B=300, T=2, w=0.05)]


@pytest.mark.parametrize("bn", ["32", "64", "96", "128"])
@pytest.mark.parametrize("cfg", TC_CASES)
def test_tc_recurrence_bit_exact(qnn, cfg, bn, monkeypatch):
    wl = _small(**cfg)
    params, x = wl.make()
    ref = _oracle(wl, params, x, want_h_all=True)
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    monkeypatch.setenv("QNN_TC_BN", bn)
    # the fused gate kernel takes 128/64/32-column tiles; the 96-column one serves the px path
    monkeypatch.setenv("QNN_TC_FUSE_X", "0" if bn == "96" else "1")
    qnn.profile_read()
    qnn.profile_enable(True)
    got = _gpu_forward(qnn, wl, params, x)
    qnn.profile_enable(False)
    kernels = qnn.profile_read()
    assert "lstm_gates_tc" in kernels and "lstm_recurrent" not in kernels, kernels
    _compare(got, ref, wl, params)


@pytest.mark.parametrize("fuse", ["1", "0"])
@pytest.mark.parametrize("cfg", [dict(L=2, I=40, H=100, C=37, B=130, T=4), dict(L=2, I=80, H=1100, P=64, C=20, B=40, T=3,
                                                                                 w=0.05),
                                 dict(L=2, I=600, H=64, P=48, B=70, T=3)])
def test_tc_input_product_fused_and_batched(qnn, cfg, fuse, monkeypatch):
    # the step's input product computed inside the gate kernel (default) and by the batched product
    # (QNN_TC_FUSE_X=0) give the oracle's results bit for bit; I = 600 puts the input on two
    # chunk-sized parts of the fused K loop (10 k-blocks of x, then those of h)
    wl = _small(**cfg)
    params, x = wl.make()
    ref = _oracle(wl, params, x, want_h_all=True)
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    monkeypatch.setenv("QNN_TC_FUSE_X", fuse)
    got = _gpu_forward(qnn, wl, params, x)
    _compare(got, ref, wl, params)


# The LSTMP projection of a step in both of its forms, split-K partial sums with a finishing row
# kernel (the default) and one product whose epilogue writes r_t (QNN_TC_PROJ=linear), against the
# oracle: a partial last 128-row block, a projection wider than the cells (H = 100, P = 256), two
# exact accumulation chunks with a short second one (H = 1100), and the full 2048 x 512 shape.
PROJ_CASES = [dict(L=2, I=40, H=256, P=128, C=11, B=130, T=4, w=0.1),
              dict(L=1, I=24, H=100, P=256, B=64, T=3),
              dict(L=1, I=16, H=1100, P=384, B=70, T=3, w=0.1),
              dict(L=2, I=80, H=2048, P=512, C=20, B=129, T=3, w=0.05)]


@pytest.mark.parametrize("mode", ["split", "linear"])
@pytest.mark.parametrize("cfg", PROJ_CASES)
def test_tc_lstmp_projection_forms(qnn, cfg, mode, monkeypatch):
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    monkeypatch.setenv("QNN_TC_PROJ", mode)
    wl = _small(**cfg)
    params, x = wl.make()
    ref = _oracle(wl, params, x, want_h_all=True)
    qnn.profile_read()
    qnn.profile_enable(True)
    got = _gpu_forward(qnn, wl, params, x)
    qnn.profile_enable(False)
    kernels = qnn.profile_read()
    assert ("proj_finish" in kernels) == (mode == "split"), kernels
    _compare(got, ref, wl, params)


# The layers as a wavefront across streams (the kernel that quantizes a step's outputs for the
# layer's next step also writes the next layer's input codes of the step; QNN_TC_WAVE=0 runs the
# layers one after the other): the oracle's results bit for bit, with carried state in and out,
# with the layer outputs requested (kept whole for every layer) and without (only the top layer's),
# and equal to the sequential schedule; LSTMP with the split and the linear projection, and LSTM.
@pytest.mark.parametrize("want_h_all", [True, False])
@pytest.mark.parametrize("proj", ["split", "linear", "none"])
def test_tc_layer_wavefront(qnn, want_h_all, proj, monkeypatch):
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    monkeypatch.setenv("QNN_TC_PROJ", "linear" if proj == "linear" else "split")
    wl = _small(L=3, I=40, H=256, P=0 if proj == "none" else 128, C=13, B=130, T=5, w=0.1)
    params, x = wl.make()
    g = rng(77)
    h0 = g.uniform(-0.5, 0.5, (wl.num_layers, wl.batch, wl.R)).astype(np.float32)
    c0 = g.uniform(-1.0, 1.0, (wl.num_layers, wl.batch, wl.hidden)).astype(np.float32)
    ref = _oracle(wl, params, x, want_h_all=True, h0=h0, c0=c0)
    outs = {}
    for wave in ("1", "0"):
        monkeypatch.setenv("QNN_TC_WAVE", wave)
        got = _gpu_forward(qnn, wl, params, x, h_all=want_h_all, h0=h0, c0=c0)
        _compare(got, ref, wl, params)  # (h_all compared when requested)
        outs[wave] = got
    for k in ("y", "h", "c", "logits"):
        assert np.array_equal(outs["1"][k], outs["0"][k]), k


# The wavefront's own launch shapes (gate grid below one block per SM, whole tiles in the last wave,
# the projection in the fewest exact K ranges) on a batch of 3 row tiles and 64 column tiles: 192
# tiles on 136 blocks, so blocks take a second tile of another row tile (their per-row constants
# recomputed). Equal to the layers run in sequence bit for bit, and to the oracle on one sequence
# of each row tile.
def test_tc_wavefront_shapes_row_tile_changes(qnn, monkeypatch):
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    wl = _small(L=2, I=80, H=2048, P=256, C=37, B=384, T=4, w=0.05, wo=0.5)
    params, x = wl.make()
    outs = {}
    for wave in ("1", "0"):
        monkeypatch.setenv("QNN_TC_WAVE", wave)
        outs[wave] = _gpu_forward(qnn, wl, params, x, h_all=False)
    for k in ("y", "h", "c", "logits"):
        assert np.array_equal(outs["1"][k], outs["0"][k]), k
    seqs = (0, 200, 383)
    for b, ref in zip(seqs, _sequences_by_oracle(wl, params, x, seqs)):
        _check_sequence(outs["1"], ref, b)


# The 8-bit output layer beside the recurrence (wavefront): chunks of frames as the top layer
# completes them, from the codes its step kernels write, logits time-major and the softmax into the
# sequence-major posteriors. Chunks of 1 and 2 frames (a short last chunk) and one chunk, LSTM and
# LSTMP; logits bit-exact, and everything equal to the output layer run after the recurrence.
@pytest.mark.parametrize("chunk", ["1", "2", ""])
@pytest.mark.parametrize("P", [0, 128])
def test_tc_output_layer_beside_recurrence(qnn, chunk, P, monkeypatch):
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    if chunk:
        monkeypatch.setenv("QNN_OUT_CHUNK", chunk)
    wl = _small(L=2, I=40, H=256, P=P, C=37, B=130, T=5, w=0.1, wo=0.5)
    params, x = wl.make()
    ref = _oracle(wl, params, x, want_h_all=True)
    outs = {}
    for ov in ("1", "0"):
        monkeypatch.setenv("QNN_OUT_OVERLAP", ov)
        got = _gpu_forward(qnn, wl, params, x)
        _compare(got, ref, wl, params)
        outs[ov] = got
    for k in ("y", "logits", "h", "c"):
        assert np.array_equal(outs["1"][k], outs["0"][k]), k


# posteriors for pinned host memory: staged in two device buffers of a chunk and copied out
# beside the recurrence (chunks of 1, 2 and 3 frames of 5: buffers reused, a ragged last chunk), or
# written to the host by the softmax itself; both equal the device-memory result
@pytest.mark.parametrize("stage", ["1", "0"])
@pytest.mark.parametrize("chunk", ["1", "2", "3"])
def test_tc_output_posteriors_to_pinned_host(qnn, chunk, stage, monkeypatch):
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    monkeypatch.setenv("QNN_OUT_CHUNK", chunk)
    monkeypatch.setenv("QNN_OUT_STAGE", stage)
    wl = _small(L=2, I=40, H=256, P=64, C=37, B=130, T=5, w=0.1, wo=0.5)
    params, x = wl.make()
    ref = _oracle(wl, params, x)
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode)
    model = qnn.LstmModel(d, gpu(params))
    y_dev = model.forward(gpu(x)).cpu().numpy()
    x_host = torch.from_numpy(x).pin_memory()
    y_host = torch.full((wl.batch, wl.frames, wl.num_classes), float("nan"), dtype=torch.float32).pin_memory()
    for _ in range(2):  # the second pass reuses the staging buffers
        model.forward(x_host, y=y_host)
        torch.cuda.synchronize()
        assert qnn.device_status() == qnn.QNN_OK
        assert np.array_equal(y_host.numpy(), y_dev)
    parity.check_posteriors(y_dev, ref["y"])


# 192 tiles of the gate product on 152 SMs: the 40 tiles of the last wave run as 80 half-width
# items (N = 64 or 32); the same results with whole tiles (QNN_TC_HALF=0) and from the oracle
@pytest.mark.parametrize("half", ["1", "0"])
@pytest.mark.parametrize("bn,cfg", [("128", dict(L=1, I=40, H=2048, P=128, B=384, T=2, w=0.05)),
                                    ("64", dict(L=1, I=40, H=1024, B=384, T=2, w=0.05))])
def test_tc_last_wave_half_tiles(qnn, bn, cfg, half, monkeypatch):
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    monkeypatch.setenv("QNN_TC_BN", bn)
    monkeypatch.setenv("QNN_TC_HALF", half)
    wl = _small(**cfg)
    params, x = wl.make()
    ref = _oracle(wl, params, x, want_h_all=True)
    got = _gpu_forward(qnn, wl, params, x)
    _compare(got, ref, wl, params)


@pytest.mark.parametrize("bn,fuse", [("32", "1"), ("64", "1"), ("96", "0")])
def test_tc_recurrence_large_weight_offsets(qnn, bn, fuse, monkeypatch):
    # every weight shifted by +20: weight ranges far from zero give offsets z of about 32000, so
    # K |a' + za| |w' + zw| exceeds 2^31 and the gate epilogue sums S in 64 bits
    wl = _small(L=1, I=40, H=128, B=70, T=3, w=0.08)
    params, x = wl.make()
    params = (params + np.float32(20.0)).astype(np.float32)
    ref = _oracle(wl, params, x, want_h_all=True)
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    monkeypatch.setenv("QNN_TC_BN", bn)
    monkeypatch.setenv("QNN_TC_FUSE_X", fuse)
    got = _gpu_forward(qnn, wl, params, x)
    _compare(got, ref, wl, params)


def test_tc_recurrence_state_round_trip(qnn, monkeypatch):
    """Streaming: two calls on halves of the frames give the single call's outputs and state."""
    monkeypatch.setenv("QNN_LSTM_PATH", "tc")
    wl = _small(L=2, I=12, H=68, P=20, C=0, B=70, T=8)
    params, x = wl.make()
    ref = _oracle(wl, params, x, want_h_all=True)
    first = _gpu_forward(qnn, wl, params, x[:, :3])
    second = _gpu_forward(qnn, wl, params, x[:, 3:], h0=first["h"], c0=first["c"])
    assert np.array_equal(np.concatenate([first["h_all"], second["h_all"]], axis=2), ref["h_all"])
    assert np.array_equal(second["h"], ref["h"]) and np.array_equal(second["c"], ref["c"])


def test_large_batches_take_the_tc_path(qnn, monkeypatch):
    monkeypatch.delenv("QNN_LSTM_PATH", raising=False)
    monkeypatch.delenv("QNN_TC_BN", raising=False)
    for B, want in ((63, False), (64, True)):
        wl = _small(L=1, I=8, H=32, B=B, T=2)
        params, x = wl.make()
        qnn.profile_read()
        qnn.profile_enable(True)
        got = _gpu_forward(qnn, wl, params, x)
        qnn.profile_enable(False)
        assert ("lstm_gates_tc" in qnn.profile_read()) == want
        _compare(got, _oracle(wl, params, x, want_h_all=True), wl)


def test_benchmarked_workload_takes_the_small_path(qnn, monkeypatch):
    monkeypatch.delenv("QNN_LSTM_PATH", raising=False)
    wl = inputs.LSTM_5x500_B1
    params, x = wl.make(frames=8)
    qnn.profile_read()
    qnn.profile_enable(True)
    _gpu_forward(qnn, wl, params, x, h_all=False)
    qnn.profile_enable(False)
    assert "lstm_small" in qnn.profile_read()


# ------------------------------------------------------------------------------------------
# Frame stacking (Sec. 4 frontend)
# ------------------------------------------------------------------------------------------

@pytest.mark.parametrize("B,T,I,n,stride", [(1, 300, 40, 8, 3), (3, 17, 40, 8, 3), (2, 5, 7, 3, 2), (4, 1, 12, 8, 3),
                                            (2, 50, 80, 1, 1), (5, 31, 3, 4, 5)])
def test_stack_frames_bit_exact(qnn, B, T, I, n, stride):
    x = rng(B * 1000 + T + I).normal(0, 1, (B, T, I)).astype(np.float32)
    got = qnn.stack_frames(gpu(x), n, stride)
    assert qnn.device_status() == qnn.QNN_OK
    assert np.array_equal(got.cpu().numpy(), oracle.stack_frames(x, n, stride))


@pytest.mark.parametrize("path,B", [("small", 2), ("layerwise", 5), ("tc", 70)])
def test_lstm_with_stacked_frames(qnn, path, B, monkeypatch):
    """A model with the paper's frontend (8 frames of 40 features, every third presented) against the
    oracle run on the stacked frames; raw frames passed as device memory and as host memory."""
    monkeypatch.setenv("QNN_LSTM_PATH", path)
    L, I, H, C, T, n, stride = 2, 40, 64, 11, 20, 8, 3
    wl = _small(L=L, I=I * n, H=H, C=C, B=B, T=T, w=0.1)
    params, _ = wl.make()
    x = rng(B + 7).normal(0, 1, (B, T, I)).astype(np.float32)
    xs = oracle.stack_frames(x, n, stride)
    ref = _oracle(wl, params, xs, want_h_all=True)
    d = qnn.lstm_desc(L, I, H, 0, C, stack=n, stack_stride=stride)
    model = qnn.LstmModel(d, gpu(params))
    Tp = xs.shape[1]
    ha = torch.empty((L, B, Tp, H), dtype=torch.float32, device="cuda")
    hs = torch.zeros((L, B, H), dtype=torch.float32, device="cuda")
    cs = torch.zeros((L, B, H), dtype=torch.float32, device="cuda")
    lg = torch.empty((B, Tp, C), dtype=torch.float32, device="cuda")
    y = model.forward(gpu(x), h_state=hs, c_state=cs, h_all=ha, logits=lg)
    assert qnn.device_status() == qnn.QNN_OK
    assert y.shape == (B, Tp, C)
    got = {"y": y.cpu().numpy(), "h": hs.cpu().numpy(), "c": cs.cpu().numpy(), "h_all": ha.cpu().numpy(),
           "logits": lg.cpu().numpy()}
    _compare(got, ref, wl, params)
    y_host = model.forward(x)  # host frames: staged inside the call
    assert np.array_equal(y_host, got["y"])


# ------------------------------------------------------------------------------------------
# Sub-matrix granularity (Sec. 3.1): every weight matrix as equal row blocks, each its own unit
# ------------------------------------------------------------------------------------------

def _block_scaled(params, wl, nb, seed):
    """Rescale the row blocks of every weight matrix by different factors, so that a lookup of the
    wrong block's unit shows."""
    H, P, R = wl.hidden, wl.proj, wl.R
    f = rng(seed).choice([0.05, 0.3, 1.0, 4.0], size=nb).astype(np.float32)
    p = params.copy()
    off = 0

    def scale(rows, cols):
        nonlocal off
        blk = p[off:off + rows * cols].reshape(nb, rows // nb, cols)
        blk *= f[:, None, None]
        off += rows * cols

    for l in range(wl.num_layers):
        for _ in range(4):
            scale(H, wl.layer_in(l))
        for _ in range(4):
            scale(H, R)
        off += 4 * H
        if P > 0:
            scale(P, H)
    if wl.num_classes > 0:
        scale(wl.num_classes, R)
    return p


SUB_CASES = [("small", dict(L=2, I=40, H=96, C=12, B=2, T=10), 4), ("layerwise", dict(L=2, I=24, H=48, P=16, C=8, B=9, T=5), 2),
             ("tc", dict(L=2, I=24, H=64, P=32, C=16, B=70, T=4), 4), ("tc", dict(L=1, I=40, H=96, B=130, T=3), 3),
             ("tc", dict(L=2, I=24, H=128, P=128, C=16, B=70, T=4), 4),
             ("layerwise", dict(L=1, I=40, H=12, B=6, T=5), 6)]


@pytest.mark.parametrize("path,cfg,nb", SUB_CASES)
def test_lstm_sub_matrix_units_bit_exact(qnn, path, cfg, nb, monkeypatch):
    monkeypatch.setenv("QNN_LSTM_PATH", path)
    wl = _small(**cfg)
    params, x = wl.make()
    params = _block_scaled(params, wl, nb, seed=nb)
    od = oracle.desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode, nb)
    ref = oracle.lstm_forward(od, params, x, want_h_all=True, want_logits=wl.num_classes > 0)
    d = qnn.lstm_desc(wl.num_layers, wl.input_dim, wl.hidden, wl.proj, wl.num_classes, wl.output_mode,
                      weight_blocks=nb)
    model = qnn.LstmModel(d, gpu(params))
    B, T, _ = x.shape
    ha = torch.empty((wl.num_layers, B, T, wl.R), dtype=torch.float32, device="cuda")
    hs = torch.zeros((wl.num_layers, B, wl.R), dtype=torch.float32, device="cuda")
    cs = torch.zeros((wl.num_layers, B, wl.hidden), dtype=torch.float32, device="cuda")
    lg = torch.empty((B, T, wl.num_classes), dtype=torch.float32, device="cuda") if wl.num_classes else None
    qnn.profile_read()
    qnn.profile_enable(True)
    y = model.forward(gpu(x), h_state=hs, c_state=cs, h_all=ha, logits=lg)
    qnn.profile_enable(False)
    kernels = qnn.profile_read()
    want = {"small": "lstm_small", "tc": "lstm_gates_tc", "layerwise": "lstm_recurrent"}[path]
    assert want in kernels, kernels
    assert qnn.device_status() == qnn.QNN_OK
    got = {"y": y.cpu().numpy(), "h": hs.cpu().numpy(), "c": cs.cpu().numpy(), "h_all": ha.cpu().numpy()}
    if lg is not None:
        got["logits"] = lg.cpu().numpy()
    _compare(got, ref, wl, params)
    codes, prm = model.weights()
    c_ref, p_ref = oracle.lstm_quantize_weights(od, params)
    assert np.array_equal(codes, c_ref) and np.array_equal(prm.view(np.int32), p_ref.view(np.int32))


def test_sub_matrix_units_must_divide_the_rows(qnn):
    d = qnn.lstm_desc(1, 8, 12, 0, 0, weight_blocks=5)  # 12 rows per gate matrix do not split in 5
    assert qnn.qnn_lstm_param_count(d) == -1
    h = ctypes.c_void_p()
    params = torch.zeros(qnn.qnn_lstm_param_count(qnn.lstm_desc(1, 8, 12)), device="cuda")
    assert qnn.lib().qnn_lstm_model_create(ctypes.byref(d), ctypes.c_void_p(params.data_ptr()),
                                           ctypes.byref(h)) == qnn.QNN_ERR_INVALID_ARG
