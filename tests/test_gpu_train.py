"""The AdamW update kernel against the oracle, and the full training step of
the 3-layer dense SNN (forward, loss, BPTT, AdamW) through the C ABI."""
import numpy as np
import pytest
import torch

from oracle import snn_oracle as O
from paper_2211_10725_gb300 import snn
from paper_2211_10725_gb300 import workloads as W
from paper_2211_10725_gb300.dsnn import DenseSNN
from tests import scan_harness as H

pytestmark = pytest.mark.gpu

HYPER = dict(lr=1e-2, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.05)


def _f32(x):
    return float(np.float32(x))


def _adam_tol(w_ref, m_mag, v_ref, step, lr, beta1, beta2, eps):
    """fp32 evaluation of one update: at most 16 roundings on each of w's
    two terms (the decayed weight; the Adam step, lr times the bias-corrected
    ratio, whose bias corrections the kernel may evaluate in float), where
    the first moment's own error is judged against the magnitude of the
    terms it sums (m_mag)."""
    ratio = (m_mag / (1 - beta1 ** step)) / (np.sqrt(v_ref / (1 - beta2 ** step)) + eps)
    return 16 * H.EPS32 * (np.abs(w_ref) + lr * ratio) + 1e-30


@pytest.mark.parametrize("n", [1, 7, 4096, 1001, 1 << 20])
@pytest.mark.parametrize("use_counter", [False, True])
def test_adamw_matches_oracle(n, use_counter, cuda_device):
    g = torch.Generator().manual_seed(n)
    w0 = torch.randn(n, generator=g, dtype=torch.float32)
    h = {k: _f32(v) for k, v in HYPER.items()}
    w, m, v = (w0.double().numpy(), np.zeros(n), np.zeros(n))
    m_mag = np.zeros(n)
    dw = w0.to(cuda_device)
    dm = torch.zeros(n, device=cuda_device)
    dv = torch.zeros(n, device=cuda_device)
    dlow = torch.empty(n, dtype=torch.bfloat16, device=cuda_device)
    counter = torch.zeros(2, dtype=torch.int64, device=cuda_device) if use_counter else None
    for step in (1, 2, 3):
        grad = torch.randn(n, generator=g, dtype=torch.float32) * (10.0 ** (step - 2))
        snn.snn_adamw_step(dw, dlow, grad.to(cuda_device), dm, dv, h["lr"], h["beta1"],
                           h["beta2"], h["eps"], h["weight_decay"], step=step,
                           step_counter=counter)
        torch.cuda.synchronize()
        w, m, v = O.adamw_step(w, grad.double().numpy(), m, v, h["lr"], h["beta1"], h["beta2"],
                               h["eps"], h["weight_decay"], step)
        m_mag = h["beta1"] * m_mag + (1 - h["beta1"]) * np.abs(grad.double().numpy())
        tol = _adam_tol(w, m_mag, v, step, h["lr"], h["beta1"], h["beta2"], h["eps"]) * step
        H.assert_close(f"w step {step}", dw.cpu().double().numpy(), w, 0.0, tol)
        H.assert_close(f"m step {step}", dm.cpu().double().numpy(), m, 4 * H.EPS32 * step, 0.0,
                       m_mag)
        H.assert_close(f"v step {step}", dv.cpu().double().numpy(), v, 4 * H.EPS32 * step, 0.0)
        assert torch.equal(dlow.cpu(), dw.cpu().to(torch.bfloat16))
    if use_counter:
        assert counter.cpu().tolist() == [3, 0]


def test_adamw_argument_checks(cuda_device):
    lib = snn.load_library()
    w = torch.zeros(64, device=cuda_device)
    p = w.data_ptr()
    args = (0.01, 0.9, 0.999, 1e-8, 0.0)
    assert lib.snn_adamw_step(0, None, None, None, None, None, *args, 1, None, None) == 0
    assert lib.snn_adamw_step(8, p, None, p, p, p, *args, 0, None, None) == 1      # step < 1
    assert lib.snn_adamw_step(8, p + 4, None, p, p, p, *args, 1, None, None) == 2  # alignment
    assert lib.snn_adamw_step(8, p, None, p, p, p, 0.01, 1.0, 0.999, 1e-8, 0.0, 1, None,
                              None) == 1                                          # beta1


def test_dsnn_training_lowers_the_loss(cuda_device):
    """Full training steps on one fixed batch of the 784-1000-1000-10 T=25
    B=128 network: the first update moves no weight by more than lr (Adam's
    bias-corrected first step has |m_hat| / sqrt(v_hat) <= 1) beyond the
    decay, the device step counter advances, and the loss falls."""
    w = W.DSNN_C3
    inp = W.make_dense_inputs(w)
    net = DenseSNN(w, inp["W"], device=cuda_device, lr=2e-3)
    X = inp["X"].reshape(w.T * w.B, -1).to(cuda_device)
    labels = inp["labels"].to(cuda_device)
    w_before = net.W32_flat.clone()
    losses = [float(net.train_step(X, labels).item())]
    torch.cuda.synchronize()
    moved = (net.W32_flat - w_before * (1 - net.lr * net.weight_decay)).abs().max().item()
    assert moved <= net.lr * (1 + 1e-4)
    assert torch.equal(net.W_flat.cpu(), net.W32_flat.cpu().to(torch.bfloat16))
    for _ in range(29):
        losses.append(float(net.train_step(X, labels).item()))
    torch.cuda.synchronize()
    assert net.step_counter.cpu().tolist() == [30, 0]
    for layer in net.layers:
        assert layer.status() == 0
    assert np.all(np.isfinite(losses))
    assert min(losses[-5:]) < 0.8 * losses[0], losses


def _net(kind, save, device):
    if kind == "dsnn":
        w = W.DSNN_C3
        inp = W.make_dense_inputs(w)
        net = DenseSNN(w, inp["W"], device=device, save=save, lr=2e-3)
        X = inp["X"].reshape(w.T * w.B, -1).to(device)
    else:
        from paper_2211_10725_gb300.csnn import ConvSNN
        w = W.CSNN_C4
        inp = W.make_conv_inputs(w)
        net = ConvSNN(w, inp["convs"], inp["Wfc"], device=device, save=save)
        X = inp["X"].reshape(w.T * w.B, w.H, w.W, w.Cin).to(device)
    return net, X, inp["labels"].to(device)


def _state(net):
    out = [net.loss, net.W32_flat, net.W_flat, net.m_flat, net.v_flat, net.dW_flat]
    for name in ("beta_flat", "dbeta_flat"):
        if getattr(net, name, None) is not None:
            out.append(getattr(net, name))
    return [t.detach().clone() for t in out]


@pytest.mark.parametrize("kind,save", [("dsnn", "fused"), ("dsnn", "mem"), ("csnn", "fused")])
def test_side_stream_step_is_bit_identical(kind, save, cuda_device):
    """Three training steps with the weight gradients forked onto a second
    stream (eagerly, then replayed from a captured CUDA graph) leave every
    weight, moment, gradient and the loss bit for bit as the same steps with
    every launch in line on one stream: the fork moves launches, not
    arithmetic."""
    ref, X, labels = _net(kind, save, cuda_device)
    for _ in range(3):
        ref.train_step(X, labels)
    torch.cuda.synchronize()
    want = _state(ref)

    net, X, labels = _net(kind, save, cuda_device)
    side = snn.SideStream(cuda_device)
    net.train_step(X, labels, side=side)
    stream = torch.cuda.Stream(cuda_device)
    stream.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    # the capture records the second step's launches; the step counter
    # lives on the device, so each replay is the next step
    with torch.cuda.graph(g, stream=stream):
        net.train_step(X, labels, stream=None, side=side)
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    for a, b in zip(_state(net), want):
        assert torch.equal(a, b)
