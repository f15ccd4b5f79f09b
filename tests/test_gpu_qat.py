"""Quantization-aware training (Algorithm 1) for fully connected layers: the forward pass is the
quantized inference of Sec. 3.1 (bit for bit the oracle's), the backward pass is full precision on
the float weights and on the layer input of the quantized forward pass."""
import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qat():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1607_04683_gb300 import build, qnn, qat as q
    build.build()
    qnn.lib()
    torch.cuda.set_device(0)
    torch.backends.cuda.matmul.allow_tf32 = False
    return q


def _layer(q, K, N, nb, seed):
    g = np.random.Generator(np.random.PCG64(seed))
    layer = q.QuantLinear(K, N, n_blocks=nb)
    with torch.no_grad():
        layer.weight.copy_(torch.from_numpy(g.uniform(-0.2, 0.2, (N, K)).astype(np.float32)))
        layer.bias.copy_(torch.from_numpy(g.normal(0, 0.1, N).astype(np.float32)))
    x = g.normal(0, 1, (33, K)).astype(np.float32)
    return layer, x, g


@pytest.mark.parametrize("K,N,nb", [(40, 24, 1), (300, 128, 4), (512, 200, 1)])
def test_forward_is_quantized_inference(qat, K, N, nb):
    layer, x, _ = _layer(qat, K, N, nb, K + N)
    y = layer(torch.from_numpy(x).cuda())
    W = layer.weight.detach().cpu().numpy()
    ca, pa, _ = oracle.quantize(x, oracle.PER_ROW)
    parts = [oracle.quantize(w, oracle.PER_MATRIX) for w in np.split(W, nb)]
    cw = np.concatenate([p[0] for p in parts])
    pw = np.concatenate([p[1] for p in parts])
    ref = oracle.qmatmul(ca, pa, 1, cw, pw, n_blocks=nb, bias=layer.bias.detach().cpu().numpy())
    assert np.array_equal(y.detach().cpu().numpy(), ref["y"])


def test_backward_is_full_precision(qat):
    """Algorithm 1: error() through the float weights, wgradient() with the layer's float input,
    bgradient() the summed error; the quantized values never enter the gradients."""
    layer, x, g = _layer(qat, 96, 40, 1, 5)
    xt = torch.from_numpy(x).cuda().requires_grad_(True)
    y = layer(xt)
    gy = g.normal(0, 1, y.shape).astype(np.float32)
    y.backward(torch.from_numpy(gy).cuda())
    W = layer.weight.detach().cpu().numpy().astype(np.float64)
    gy64, x64 = gy.astype(np.float64), x.astype(np.float64)
    np.testing.assert_allclose(xt.grad.cpu().numpy(), gy64 @ W, rtol=1e-5, atol=1e-5)
    np.testing.assert_allclose(layer.weight.grad.cpu().numpy(), gy64.T @ x64, rtol=1e-5, atol=1e-5)
    np.testing.assert_allclose(layer.bias.grad.cpu().numpy(), gy64.sum(0), rtol=1e-5, atol=1e-5)
    # the recovered quantized input differs from x by up to half a step: a straight-through
    # estimator built on it would give a measurably different weight gradient
    ca, pa, _ = oracle.quantize(x, oracle.PER_ROW)
    xq = np.stack([oracle.recover(ca[i], pa[i]) for i in range(len(x))]).astype(np.float64)
    assert np.abs(gy64.T @ xq - gy64.T @ x64).max() > 100 * 1e-5 * np.abs(gy64.T @ x64).max()


def test_training_reduces_the_loss(qat):
    """A two-layer softmax classifier on synthetic data (labels from a random teacher) trained by
    Algorithm 1 ("quant-all"): quantized forward, full-precision SGD updates."""
    torch.manual_seed(0)
    g = np.random.Generator(np.random.PCG64(9))
    K, Hd, C, M = 40, 64, 8, 512
    X = torch.from_numpy(g.normal(0, 1, (M, K)).astype(np.float32)).cuda()
    teacher = torch.from_numpy(g.normal(0, 1, (K, C)).astype(np.float32)).cuda()
    labels = (X @ teacher).argmax(1)
    l1, l2 = qat.QuantLinear(K, Hd), qat.QuantLinear(Hd, C)
    opt = torch.optim.SGD(list(l1.parameters()) + list(l2.parameters()), lr=0.5)

    def loss_fn():
        return torch.nn.functional.cross_entropy(l2(torch.tanh(l1(X))), labels)

    first = float(loss_fn().detach())
    for _ in range(150):
        opt.zero_grad()
        loss = loss_fn()
        loss.backward()
        opt.step()
    last = float(loss_fn().detach())
    assert last < 0.5 * first, (first, last)
