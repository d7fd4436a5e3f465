"""Parity of the tcgen05 dense-layer GEMM and the rate-coded loss with the
CPU oracle (through the C ABI)."""
import numpy as np
import pytest
import torch

from oracle import snn_oracle as O
from paper_2211_10725_gb300 import snn
from paper_2211_10725_gb300 import workloads as W
from tests import scan_harness as H

pytestmark = pytest.mark.gpu


def _bf16(shape, seed, scale=1.0, spikes=False):
    g = torch.Generator().manual_seed(seed)
    if spikes:
        return (torch.rand(shape, generator=g) < 0.2).to(torch.bfloat16)
    return (scale * torch.randn(shape, generator=g)).to(torch.bfloat16)


def _np(t):
    return t.float().numpy().astype(np.float64)


# (M, K, N): tile-aligned, ragged, the 3-layer network's forward and backward shapes
SHAPES = [(128, 64, 128), (200, 72, 40), (136, 16, 1000), (3200, 784, 1000),
          (3200, 1000, 16), (3200, 16, 1000), (1000, 3200, 784), (16, 3200, 1000),
          (200, 576, 300), (4096, 2048, 1024)]


@pytest.mark.parametrize("M,K,N", SHAPES)
def test_dense_forward(M, K, N, cuda_device):
    X = _bf16((M, K), M + K, spikes=True)
    Wt = _bf16((N, K), N + 7, scale=(6.0 / K) ** 0.5)
    ws = torch.zeros(256, dtype=torch.uint8, device=cuda_device)
    I = torch.full((M, N), float("nan"), dtype=torch.float32, device=cuda_device)
    snn.snn_dense_layer_fwd(X.to(cuda_device), Wt.to(cuda_device), I, ws)
    torch.cuda.synchronize()
    ref = O.dense_forward(_np(X), _np(Wt))
    scale = np.abs(_np(X)) @ np.abs(_np(Wt)).T   # magnitude of the summed terms
    H.assert_close("I", I.cpu().numpy(), ref, 1e-5, 1e-6, scale)


@pytest.mark.parametrize("M,K,N", [(128, 64, 128), (200, 72, 40), (3200, 784, 1000),
                                   (3200, 1000, 16), (3200, 1000, 1000), (136, 16, 1000),
                                   (2048, 512, 256)])
def test_dense_backward(M, K, N, cuda_device):
    X = _bf16((M, K), M, spikes=True)
    Wt = _bf16((N, K), N, scale=(6.0 / K) ** 0.5)
    dI = _bf16((M, N), M + N, scale=1e-2)
    ws = torch.zeros(snn.snn_dense_workspace_bytes(M, K, N), dtype=torch.uint8, device=cuda_device)
    dX = torch.full((M, K), float("nan"), dtype=torch.bfloat16, device=cuda_device)
    dW = torch.full((N, K), float("nan"), dtype=torch.float32, device=cuda_device)
    d = lambda t: t.to(cuda_device)
    snn.snn_dense_layer_bwd(d(X), d(Wt), d(dI), dX, dW, ws)
    torch.cuda.synchronize()
    rdX, rdW = O.dense_backward(_np(X), _np(Wt), _np(dI))
    sdX = np.abs(_np(dI)) @ np.abs(_np(Wt))
    sdW = np.abs(_np(dI)).T @ np.abs(_np(X))
    H.assert_close("dX", _np(dX.cpu()), rdX, 2 ** -8, 1e-6, np.maximum(np.abs(rdX), 1e-5 * sdX))
    H.assert_close("dW", dW.cpu().numpy(), rdW, 1e-5, 1e-6, sdW)


def test_dense_argument_checks(cuda_device):
    lib = snn.load_library()
    assert lib.snn_dense_layer_fwd(8, 12, 8, 16, 16, 16, 16, 256, None) == 3   # K % 8
    assert lib.snn_dense_layer_fwd(8, 16, 8, 16, 24, 16, 16, 256, None) == 2   # alignment
    assert lib.snn_dense_layer_fwd(8, 16, 8, 16, 16, 16, 16, 64, None) == 4    # workspace
    assert lib.snn_dense_layer_bwd(8, 16, 10, 16, 16, 16, 16, 16, 16, 1 << 20, None) == 3


# (T, B, C, ld): the 3-layer network's readout; more classes than a warp's
# lanes with samples in several shared-memory chunks; the largest class count
@pytest.mark.parametrize("T,B,C,ld", [(25, 128, 10, 16), (7, 300, 100, 104), (3, 20, 1024, 1032),
                                      (1, 1, 1, 8)])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_rate_ce_loss(T, B, C, ld, dtype, cuda_device):
    g = torch.Generator().manual_seed(3 + B)
    spk = (torch.rand((T, B, ld), generator=g) < 0.3).to(dtype)
    labels = torch.randint(0, C, (B,), generator=g, dtype=torch.int32)
    loss = torch.zeros(1, dtype=torch.float32, device=cuda_device)
    grad = torch.full((T, B, ld), float("nan"), dtype=dtype, device=cuda_device)
    snn.snn_rate_ce_loss(spk.to(cuda_device), labels.to(cuda_device), C, loss, grad)
    torch.cuda.synchronize()
    rl, rg = O.rate_ce_loss(_np(spk[:, :, :C]), labels.numpy())
    assert abs(loss.item() - rl) <= 1e-6 * max(1.0, abs(rl))
    got = _np(grad.cpu())
    tol = 1e-7 if dtype == torch.float32 else 2 ** -8 * np.abs(rg).max()
    np.testing.assert_allclose(got[:, :, :C], rg, rtol=1e-5 if dtype == torch.float32 else 2e-2,
                               atol=tol)
    assert np.all(got[:, :, C:] == 0)


def test_rate_ce_loss_shard_normalisation(cuda_device):
    """A shard of a larger batch: loss and gradient are averaged over the
    global batch, so they are the shard's own values times B / batch_total."""
    T, B, C, ld, total = 25, 64, 10, 16, 256
    g = torch.Generator().manual_seed(5)
    spk = (torch.rand((T, B, ld), generator=g) < 0.3).to(torch.float32)
    labels = torch.randint(0, C, (B,), generator=g, dtype=torch.int32)
    loss = torch.zeros(1, dtype=torch.float32, device=cuda_device)
    grad = torch.full((T, B, ld), float("nan"), dtype=torch.float32, device=cuda_device)
    snn.snn_rate_ce_loss(spk.to(cuda_device), labels.to(cuda_device), C, loss, grad,
                         batch_total=total)
    torch.cuda.synchronize()
    rl, rg = O.rate_ce_loss(_np(spk[:, :, :C]), labels.numpy())
    k = B / total
    assert abs(loss.item() - rl * k) <= 1e-6 * max(1.0, abs(rl))
    np.testing.assert_allclose(_np(grad.cpu())[:, :, :C], rg * k, rtol=1e-5, atol=1e-8)
    lib = snn.load_library()
    ws = torch.zeros(snn.snn_rate_ce_workspace_bytes(B), dtype=torch.uint8, device=cuda_device)
    args = (grad.data_ptr(), labels.data_ptr(), loss.data_ptr(), grad.data_ptr(), ws.data_ptr())
    assert lib.snn_rate_ce_loss(T, B, C, 1, ld, B - 1, 0, *args, ws.numel(), None) == 1
    assert lib.snn_rate_ce_loss(T, B, C, 2, ld, 0, 0, *args, ws.numel(), None) == 1  # C*pop > ld
    assert lib.snn_rate_ce_loss(T, B, C, 1, ld, 0, 0, *args, 64, None) == 4         # workspace


# (T, B, C, pop, ld): the population-coded output layer (500 = 10 x 50,
# padded to 504), several time steps with a ragged population
@pytest.mark.parametrize("T,B,C,pop,ld", [(1, 128, 10, 50, 504), (3, 37, 13, 7, 96)])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_rate_ce_loss_population(T, B, C, pop, ld, dtype, cuda_device):
    g = torch.Generator().manual_seed(7 + pop)
    spk = (torch.rand((T, B, ld), generator=g) < 0.2).to(dtype)
    labels = torch.randint(0, C, (B,), generator=g, dtype=torch.int32)
    loss = torch.zeros(1, dtype=torch.float32, device=cuda_device)
    grad = torch.full((T, B, ld), float("nan"), dtype=dtype, device=cuda_device)
    snn.snn_rate_ce_loss(spk.to(cuda_device), labels.to(cuda_device), C, loss, grad, pop=pop)
    torch.cuda.synchronize()
    rl, rg = O.rate_ce_loss(_np(spk[:, :, :C * pop]), labels.numpy(), pop)
    assert abs(loss.item() - rl) <= 1e-6 * max(1.0, abs(rl))
    got = _np(grad.cpu())
    tol = 1e-7 if dtype == torch.float32 else 2 ** -8 * np.abs(rg).max()
    np.testing.assert_allclose(got[:, :, :C * pop], rg,
                               rtol=1e-5 if dtype == torch.float32 else 2e-2, atol=tol)
    assert np.all(got[:, :, C * pop:] == 0)
