"""The convolutional SNN (Tab. I CSNN, 12C5-MP2-64C5-MP2-10 on 28x28
input): its layout kernels (im2col, col2im, 2x2 max pooling), the split-K
weight gradient, and the whole training step against the oracle's
composition of the same steps.

Comparison protocol
-------------------
* Layout kernels move or select values: im2col, max pooling (values and
  window positions, with ties from binary spike maps) and its backward are
  compared bit for bit; col2im adds up to KH*KW bf16 values in fp32 and
  rounds once to bf16, so it is held to one bf16 rounding (2^-8 of the
  magnitude) plus fp32 summation.
* For the training step the weights are flushed to zero below 2^-7 in
  magnitude.  Every remaining bf16 weight is then a multiple of 2^-14, every
  product with a 0/1 spike too, and every partial sum the GEMMs form stays
  below 2^7 in magnitude (at most 1024 terms below 2^-3): all such sums are
  exact in fp32 in any order.  The input currents must then equal the
  oracle's float64 currents exactly, and with them the fp32 membrane trace,
  every spike, every pooled map and every window position.
* Gradients: the path rounds to bf16 the loss gradient, each layer's dL/dI,
  the readout's input gradient, the patch-row gradients and the col2im
  result; the oracle rounds at the same points except the patch rows.  Each
  rounding moves a value by at most 2^-8 of it (2^-7 when the other side
  rounded the other way); with at most eight such points between the loss
  and the deepest gradient the tolerance is 8 * 2^-7 of the magnitude of
  the summed terms (the reverse pass run on absolute values).
"""
import numpy as np
import pytest
import torch

from oracle import snn_oracle as O
from paper_2211_10725_gb300 import snn
from paper_2211_10725_gb300 import workloads as W
from paper_2211_10725_gb300.csnn import ConvSNN
from tests import scan_harness as H

pytestmark = pytest.mark.gpu

GRAD_RTOL = 8 * 2.0 ** -7
FLUSH = 2.0 ** -7

SMALL = W.CSNN_C4.scaled(name="csnn_12c5_mp2_64c5_mp2_10_T4_B8", T=4, B=8)


def _np(t):
    return t.detach().to("cpu", torch.float32).numpy().astype(np.float64)


def _bf16(a, device):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).to(device)


# ---------------------------------------------------------------------------
# Layout kernels
# ---------------------------------------------------------------------------

def _patch_rows(X, k, Kpad):
    """Patch rows of X [M, H, W, C] in (ky, kx, c) column order, zero padded
    to Kpad columns (the layout im2col writes, by slicing)."""
    M, Hh, Ww, C = X.shape
    Ho, Wo = Hh - k + 1, Ww - k + 1
    out = np.zeros((M, Ho, Wo, k, k, C))
    for ky in range(k):
        for kx in range(k):
            out[:, :, :, ky, kx, :] = X[:, ky:ky + Ho, kx:kx + Wo, :]
    rows = out.reshape(M * Ho * Wo, k * k * C)
    return np.concatenate([rows, np.zeros((rows.shape[0], Kpad - rows.shape[1]))], axis=1)


LAYOUTS = [(3, 28, 28, 1, 5, 32), (2, 12, 12, 16, 5, 400), (2, 9, 7, 3, 3, 32),
           (4, 6, 6, 8, 1, 8), (1, 5, 5, 2, 5, 56)]


@pytest.mark.parametrize("M,Hh,Ww,C,k,Kpad", LAYOUTS)
def test_im2col_layout_and_convolution(M, Hh, Ww, C, k, Kpad, cuda_device):
    g = torch.Generator().manual_seed(M * 1000 + Hh * 10 + C)
    X = torch.randn((M, Hh, Ww, C), generator=g).to(torch.bfloat16)
    Ho, Wo = Hh - k + 1, Ww - k + 1
    cols = torch.full((M * Ho * Wo, Kpad), 7.0, dtype=torch.bfloat16, device=cuda_device)
    snn.snn_im2col_nhwc(X.to(cuda_device), cols, k, k)
    torch.cuda.synchronize()
    assert np.array_equal(_np(cols), _patch_rows(_np(X), k, Kpad))
    # the patch rows times the flattened filters are the convolution
    Cout = 16
    Wc = torch.randn((Cout, k, k, C), generator=g).to(torch.bfloat16)
    Wf = torch.zeros((Cout, Kpad), dtype=torch.bfloat16)
    Wf[:, : k * k * C] = Wc.reshape(Cout, -1)
    I = torch.empty((M * Ho * Wo, Cout), dtype=torch.float32, device=cuda_device)
    ws = torch.zeros(256, dtype=torch.uint8, device=cuda_device)
    snn.snn_dense_layer_fwd(cols, Wf.to(cuda_device), I, ws)
    torch.cuda.synchronize()
    ref = O.conv2d_nhwc(_np(X), _np(Wc))
    mag = O.conv2d_nhwc(np.abs(_np(X)), np.abs(_np(Wc)))
    H.assert_close("conv", _np(I).reshape(ref.shape), ref, 1e-5, 1e-6, mag)


@pytest.mark.parametrize("M,Hh,Ww,C,k,Kpad", LAYOUTS)
def test_col2im_is_the_convolution_input_gradient(M, Hh, Ww, C, k, Kpad, cuda_device):
    g = torch.Generator().manual_seed(M * 999 + Hh * 10 + C)
    Ho, Wo = Hh - k + 1, Ww - k + 1
    K = k * k * C
    dcols = torch.randn((M * Ho * Wo, Kpad), generator=g).to(torch.bfloat16)
    dcols[:, K:] = 1e4   # padding columns must not be read
    dX = torch.empty((M, Hh, Ww, C), dtype=torch.bfloat16, device=cuda_device)
    snn.snn_col2im_nhwc(dcols.to(cuda_device), dX, k, k)
    torch.cuda.synchronize()
    d = _np(dcols)[:, :K].reshape(M, Ho, Wo, k, k, C)
    ref, mag = np.zeros((M, Hh, Ww, C)), np.zeros((M, Hh, Ww, C))
    for ky in range(k):
        for kx in range(k):
            ref[:, ky:ky + Ho, kx:kx + Wo, :] += d[:, :, :, ky, kx, :]
            mag[:, ky:ky + Ho, kx:kx + Wo, :] += np.abs(d[:, :, :, ky, kx, :])
    H.assert_close("col2im", _np(dX), ref, 2.0 ** -8 + k * k * H.EPS32, 0.0, mag)
    # with dcols = dY * W, col2im gives the oracle's convolution dX
    Cout = 8
    Wc = torch.randn((Cout, k, k, C), generator=g).to(torch.bfloat16)
    dY = torch.randn((M, Ho, Wo, Cout), generator=g).to(torch.bfloat16)
    Wf = torch.zeros((Cout, Kpad), dtype=torch.bfloat16)
    Wf[:, :K] = Wc.reshape(Cout, -1)
    rows = M * Ho * Wo
    if rows % 8 == 0:
        dc = torch.empty((rows, Kpad), dtype=torch.bfloat16, device=cuda_device)
        ws = torch.zeros(snn.snn_dense_workspace_bytes(rows, Kpad, Cout), dtype=torch.uint8,
                         device=cuda_device)
        Xdummy = torch.zeros((rows, Kpad), dtype=torch.bfloat16, device=cuda_device)
        snn.snn_dense_layer_bwd(Xdummy, Wf.to(cuda_device), dY.reshape(rows, Cout).to(cuda_device),
                                dc, None, ws)
        snn.snn_col2im_nhwc(dc, dX, k, k)
        torch.cuda.synchronize()
        ref_dX, _ = O.conv2d_nhwc_backward(np.zeros((M, Hh, Ww, C)), _np(Wc), _np(dY))
        mag_dX, _ = O.conv2d_nhwc_backward(np.zeros((M, Hh, Ww, C)), np.abs(_np(Wc)),
                                           np.abs(_np(dY)))
        H.assert_close("conv dX", _np(dX), ref_dX, 2 * 2.0 ** -8 + 1e-5, 1e-6, mag_dX)


@pytest.mark.parametrize("M,Hh,Ww,C", [(3, 24, 24, 16), (2, 8, 8, 64), (5, 2, 6, 3), (1, 4, 2, 1)])
@pytest.mark.parametrize("kind", ["spikes", "normal"])
def test_maxpool_matches_oracle(M, Hh, Ww, C, kind, cuda_device):
    g = torch.Generator().manual_seed(M * 77 + Hh + C)
    if kind == "spikes":   # many ties: the first maximum in window order wins
        X = (torch.rand((M, Hh, Ww, C), generator=g) < 0.3).to(torch.bfloat16)
    else:
        X = torch.randn((M, Hh, Ww, C), generator=g).to(torch.bfloat16)
    Y = torch.empty((M, Hh // 2, Ww // 2, C), dtype=torch.bfloat16, device=cuda_device)
    idx = torch.empty((M, Hh // 2, Ww // 2, C), dtype=torch.uint8, device=cuda_device)
    snn.snn_maxpool2_fwd_nhwc(X.to(cuda_device), Y, idx)
    dY = torch.randn(tuple(Y.shape), generator=g).to(torch.bfloat16)
    dX = torch.full((M, Hh, Ww, C), 5.0, dtype=torch.bfloat16, device=cuda_device)
    snn.snn_maxpool2_bwd_nhwc(dY.to(cuda_device), idx, dX)
    torch.cuda.synchronize()
    ref, ref_idx = O.maxpool2_nhwc(_np(X))
    assert np.array_equal(_np(Y), ref)
    assert np.array_equal(idx.cpu().numpy().astype(np.int64), ref_idx)
    assert np.array_equal(_np(dX), O.maxpool2_nhwc_backward(_np(dY), ref_idx, X.shape))


def test_layout_argument_checks(cuda_device):
    lib = snn.load_library()
    buf = torch.zeros(1 << 16, dtype=torch.bfloat16, device=cuda_device)
    p = buf.data_ptr()
    assert lib.snn_im2col_nhwc(0, 28, 28, 1, 5, 5, 32, None, None, None) == 0   # empty
    assert lib.snn_im2col_nhwc(1, 28, 28, 1, 5, 5, 30, p, p, None) == 1         # Kpad % 8
    assert lib.snn_im2col_nhwc(1, 28, 28, 1, 5, 5, 24, p, p, None) == 1         # Kpad < K
    assert lib.snn_im2col_nhwc(1, 4, 28, 1, 5, 5, 32, p, p, None) == 1          # H < KH
    assert lib.snn_im2col_nhwc(1, 8, 8, 1, 5, 5, 32, p, p + 2, None) == 2       # cols alignment
    assert lib.snn_col2im_nhwc(1, 8, 8, 1, 5, 5, 24, p, p, None) == 1
    assert lib.snn_maxpool2_fwd_nhwc(1, 7, 8, 4, p, p, p, None) == 1            # odd H
    assert lib.snn_maxpool2_bwd_nhwc(1, 8, 8, 0, p, p, p, None) == 1            # C = 0
    assert lib.snn_maxpool2_fwd_nhwc(0, 8, 8, 4, None, None, None, None) == 0


# ---------------------------------------------------------------------------
# Direct convolution with few input channels
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("M,Hh,Ww,C,Cout,k,ldw", [(5, 28, 28, 1, 16, 5, 32), (3, 9, 11, 2, 8, 3, 24),
                                                  (2, 7, 7, 1, 4, 1, 8), (700, 28, 28, 1, 16, 5, 32),
                                                  (4, 10, 13, 1, 8, 3, 16), (3, 70, 9, 1, 16, 5, 32),
                                                  (9, 28, 28, 1, 12, 5, 32), (1300, 28, 28, 1, 12, 5, 32),
                                                  (6, 12, 12, 1, 8, 3, 16)])
def test_small_conv_matches_oracle(M, Hh, Ww, C, Cout, k, ldw, cuda_device):
    """Forward currents and the weight gradient of the direct convolution
    against the oracle's convolution and its backward; the weight gradient
    is the same bits on every call.  One input channel with a 5x5 or 3x3
    filter takes the sliding-window kernels (12 channels: the CSNN's first
    layer; 700 and 1300 images: more images than blocks, so blocks sum
    several); the others, and a 70-row map (more rows than one block's
    threads), the general ones."""
    g = torch.Generator().manual_seed(M + 31 * Cout + k)
    X = (torch.rand((M, Hh, Ww, C), generator=g) < 0.3).to(torch.bfloat16)
    Wc = torch.randn((Cout, k, k, C), generator=g).to(torch.bfloat16)
    K = k * k * C
    Wt = torch.zeros((Cout, ldw), dtype=torch.bfloat16)
    Wt[:, :K] = Wc.reshape(Cout, K)
    Wt[:, K:] = 3.0   # columns past K must not be read
    Ho, Wo = Hh - k + 1, Ww - k + 1
    I = torch.empty((M, Ho, Wo, Cout), dtype=torch.float32, device=cuda_device)
    Xd = X.to(cuda_device)
    snn.snn_conv2d_small_fwd_nhwc(Xd, Wt.to(cuda_device), I, k, k)
    dI = torch.randn((M, Ho, Wo, Cout), generator=g).to(torch.bfloat16)
    dW = torch.full((Cout, ldw), 9.0, dtype=torch.float32, device=cuda_device)
    ws = torch.empty(snn.snn_conv2d_small_dw_workspace_bytes(M, Hh, Ww, C, Cout, k, k),
                     dtype=torch.uint8, device=cuda_device)
    snn.snn_conv2d_small_dw_nhwc(Xd, dI.to(cuda_device), dW, k, k, ws)
    first = dW.clone()
    snn.snn_conv2d_small_dw_nhwc(Xd, dI.to(cuda_device), dW, k, k, ws)
    torch.cuda.synchronize()
    assert torch.equal(first, dW)
    x, wc, di = _np(X), _np(Wc), _np(dI)
    ref = O.conv2d_nhwc(x, wc)
    H.assert_close("I", _np(I), ref, 1e-5, 1e-6, O.conv2d_nhwc(x, np.abs(wc)))
    _, ref_dW = O.conv2d_nhwc_backward(x, wc, di)
    _, mag = O.conv2d_nhwc_backward(x, wc, np.abs(di))
    got = _np(dW)
    H.assert_close("dW", got[:, :K].reshape(Cout, k, k, C), ref_dW, 1e-5, 1e-6, mag)
    assert not got[:, K:].any()


def test_small_conv_argument_checks(cuda_device):
    lib = snn.load_library()
    buf = torch.zeros(1 << 16, dtype=torch.float32, device=cuda_device)
    p = buf.data_ptr()
    assert lib.snn_conv2d_small_fwd_nhwc(0, 28, 28, 1, 16, 5, 5, 32, None, None, None, None) == 0
    assert lib.snn_conv2d_small_fwd_nhwc(1, 28, 28, 2, 16, 5, 5, 64, p, p, p, None) == 3  # K > 32
    assert lib.snn_conv2d_small_fwd_nhwc(1, 28, 28, 1, 20, 5, 5, 32, p, p, p, None) == 3  # Cout
    assert lib.snn_conv2d_small_fwd_nhwc(1, 28, 28, 1, 16, 5, 5, 24, p, p, p, None) == 1  # ldw < K
    assert lib.snn_conv2d_small_fwd_nhwc(1, 28, 28, 1, 16, 5, 5, 32, p, p, p + 4, None) == 2
    assert lib.snn_conv2d_small_dw_nhwc(4, 28, 28, 1, 16, 5, 5, 32, p, p, p, p, 16, None) == 4


# ---------------------------------------------------------------------------
# Split-K weight gradient
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("M,K,N", [(18432, 32, 16), (12800, 400, 64), (3200, 1024, 16),
                                   (3200, 1000, 16), (1024, 64, 8)])
def test_split_weight_gradient(M, K, N, cuda_device):
    """dW = dI^T X over many rows onto few output tiles (split K, partials
    added in split order): close to the float64 product and the same bits
    on every call."""
    g = torch.Generator().manual_seed(M + K + N)
    X = (torch.rand((M, K), generator=g) < 0.3).to(torch.bfloat16)
    dI = (torch.randn((M, N), generator=g) * 0.01).to(torch.bfloat16)
    Wt = torch.zeros((N, K), dtype=torch.bfloat16)
    ws = torch.zeros(snn.snn_dense_workspace_bytes(M, K, N), dtype=torch.uint8, device=cuda_device)
    dW = torch.empty((N, K), dtype=torch.float32, device=cuda_device)
    dX_, dI_, W_ = X.to(cuda_device), dI.to(cuda_device), Wt.to(cuda_device)
    snn.snn_dense_layer_bwd(dX_, W_, dI_, None, dW, ws)
    first = dW.clone()
    snn.snn_dense_layer_bwd(dX_, W_, dI_, None, dW, ws)
    torch.cuda.synchronize()
    assert torch.equal(first, dW)
    ref = _np(dI).T @ _np(X)
    mag = np.abs(_np(dI)).T @ np.abs(_np(X))
    H.assert_close("dW", _np(dW), ref, 1e-5, 1e-7, mag)


# ---------------------------------------------------------------------------
# The training step
# ---------------------------------------------------------------------------

def _exact_inputs(w, seed=None):
    inp = W.make_conv_inputs(w, seed)

    def flush(t):
        t = t.clone()
        t[t.float().abs() < FLUSH] = 0
        return t

    inp["convs"] = [flush(c) for c in inp["convs"]]
    inp["Wfc"] = flush(inp["Wfc"])
    return inp


def _oracle(w, inp, stored=False):
    """The oracle's forward, and its BPTT along the trace the kernels'
    backward reads: the fp32 membrane, or with ``stored`` its bf16 rounding
    (identical on both sides here, since the forward is exact)."""
    convs = [_np(c) for c in inp["convs"]]
    Wfc = _np(inp["Wfc"])
    X = _np(inp["X"]).reshape(w.T * w.B, w.H, w.W, w.Cin)
    betas = [np.full(c, w.beta) for c, _ in w.convs]
    fwd = O.csnn_forward(X, convs, Wfc, w.T, w.B, betas, w.beta_fc, w.thr, reset=w.reset,
                         dtype=np.float32)
    if stored:
        fwd = dict(fwd, mem=[O.bf16_round(m) for m in fwd["mem"]],
                   fc_mem=O.bf16_round(fwd["fc_mem"]))
    res = O.csnn_backward(fwd, convs, Wfc, _np(inp["labels"]).astype(np.int64), w.T, w.B, betas,
                          w.beta_fc, w.thr, w.sg_param, reset=w.reset, store=O.bf16_round)
    return convs, Wfc, betas, fwd, res


def _magnitudes(w, convs, Wfc, betas, fwd, g_top):
    """The reverse pass on absolute values from |dL/dspk| of the output
    layer: for each gradient the magnitude of the terms it sums (every
    coefficient of the detached zero-reset recursion is >= 0)."""
    T, B = w.T, w.B
    n = Wfc.shape[0]
    g = O.leaky_backward(fwd["fc_mem"], fwd["fc_spk"], g_top.reshape(T, B * n),
                         np.full(B * n, w.beta_fc), np.full(B * n, w.thr), reset=w.reset,
                         detach=True, sg="fast_sigmoid", sg_param=w.sg_param)
    dI_fc = g["grad_I"].reshape(T * B, n)
    d_flat, dW_fc = O.dense_backward(np.abs(fwd["fc_in"]), np.abs(Wfc), dI_fc)
    out = {"dW_fc": dW_fc, "grad_I_fc": dI_fc, "dW": [None] * len(convs),
           "grad_I": [None] * len(convs), "dbeta": [None] * len(convs)}
    d_pool = d_flat.reshape(fwd["pool"][-1].shape)
    for l in range(len(convs) - 1, -1, -1):
        shape = fwd["I"][l].shape
        _, Ho, Wo, Co = shape
        L = B * Ho * Wo * Co
        d_spk = O.maxpool2_nhwc_backward(d_pool, fwd["idx"][l], shape)
        g = O.leaky_backward(fwd["mem"][l], fwd["spk"][l], d_spk.reshape(T, L),
                             np.tile(betas[l], B * Ho * Wo), np.full(L, w.thr), reset=w.reset,
                             detach=True, sg="fast_sigmoid", sg_param=w.sg_param)
        dI = g["grad_I"]
        prev = np.concatenate([np.zeros((1, L)), np.abs(fwd["mem"][l][:-1])], axis=0)
        out["dbeta"][l] = (dI * prev).reshape(T * B * Ho * Wo, Co).sum(axis=0)
        out["grad_I"][l] = dI.reshape(T * B, Ho, Wo, Co)
        dX, dW = O.conv2d_nhwc_backward(np.abs(fwd["ins"][l]), np.abs(convs[l]),
                                        out["grad_I"][l])
        out["dW"][l] = dW
        d_pool = dX
    return out


def _run(w, inp, device, **kw):
    net = ConvSNN(w, inp["convs"], inp["Wfc"], device=device, **kw)
    X = inp["X"].reshape(w.T * w.B, w.H, w.W, w.Cin).to(device)
    labels = inp["labels"].to(device)
    return net, X, labels


def _check_step(w, net, convs, Wfc, betas, fwd, res):
    T, B = w.T, w.B
    for l, (cout, k) in enumerate(w.convs):
        g = net.geo[l]
        Ho, Wo, cp = g[5], g[6], g[3]
        if net.I[l] is not None:  # a fused layer keeps its currents on chip
            I = _np(net.I[l]).reshape(T * B, Ho, Wo, cp)
            assert np.array_equal(I[..., :cout], fwd["I"][l]), f"conv {l} currents"
            assert not I[..., cout:].any()
        if net.layers[l].mem is not None:  # the stored trace: bf16 of the exact fp32 trace
            mem = _np(net.layers[l].mem).reshape(T * B, Ho, Wo, cp)[..., :cout].reshape(T, -1)
            assert np.array_equal(mem, O.bf16_round(fwd["mem"][l])), f"conv {l} stored membrane"
        spk = _np(net.layers[l].spk).reshape(T * B, Ho, Wo, cp)
        assert np.array_equal(spk[..., :cout].reshape(T, -1), fwd["spk"][l]), f"conv {l} spikes"
        assert not spk[..., cout:].any()
        pool = _np(net.pool[l])
        assert np.array_equal(pool[..., :cout], fwd["pool"][l]), f"pool {l}"
        idx = net.idx[l].cpu().numpy().astype(np.int64)
        assert np.array_equal(idx[..., :cout], fwd["idx"][l]), f"pool {l} positions"
    n = w.n_classes
    if net.I_fc is not None:
        Ifc = _np(net.I_fc)
        assert np.array_equal(Ifc[:, :n], fwd["fc_I"]), "readout currents"
    assert np.array_equal(_np(net.out_layer.spk)[:, :, :n].reshape(T, -1), fwd["fc_spk"])

    loss = float(net.loss.item())
    assert abs(loss - res["loss"]) <= 1e-6 * max(1.0, abs(res["loss"]))
    go = _np(net.grad_out)
    H.assert_close("grad_out", go[:, :, :n], res["grad_out"], 2.0 ** -7, 0.0)
    assert not go[:, :, n:].any()
    mag = _magnitudes(w, convs, Wfc, betas, fwd, np.abs(res["grad_out"]))

    def sc(key, ref, l=None):
        m = mag[key] if l is None else mag[key][l]
        return np.maximum(m, np.abs(ref))

    gi = _np(net.out_layer.grad_I)[:, :, :n].reshape(T * B, n)
    H.assert_close("grad_I_fc", gi, res["grad_I_fc"], GRAD_RTOL, 1e-12,
                   sc("grad_I_fc", res["grad_I_fc"]))
    H.assert_close("dW_fc", _np(net.fc_weight(net.dW_flat)), res["dW_fc"], GRAD_RTOL, 1e-12,
                   sc("dW_fc", res["dW_fc"]))
    for l, (cout, k) in enumerate(w.convs):
        g = net.geo[l]
        Ho, Wo, cp = g[5], g[6], g[3]
        gI = _np(net.layers[l].grad_I).reshape(T * B, Ho, Wo, cp)
        H.assert_close(f"grad_I{l}", gI[..., :cout], res["grad_I"][l], GRAD_RTOL, 1e-12,
                       sc("grad_I", res["grad_I"][l], l))
        assert not gI[..., cout:].any()
        H.assert_close(f"dW{l}", _np(net.conv_weight(l, net.dW_flat)), res["dW"][l], GRAD_RTOL,
                       1e-12, sc("dW", res["dW"][l], l))
        db = _np(net.dbeta[l])
        H.assert_close(f"dbeta{l}", db[:cout], res["dbeta"][l], GRAD_RTOL, 1e-9,
                       sc("dbeta", res["dbeta"][l], l))
        assert not db[cout:].any()
    # padding rows and columns of every weight gradient are exactly zero
    for l in range(len(w.convs)):
        _, _, cin_p, cout_p, k, *_r, kpad = net.geo[l]
        cout = w.convs[l][0]
        cin = w.Cin if l == 0 else w.convs[l - 1][0]
        d = _np(net.dW[l])
        assert not d[cout:].any() and not d[:, k * k * cin_p:].any(), f"dW{l} padding"
        assert not d[:, : k * k * cin_p].reshape(cout_p, k, k, cin_p)[..., cin:].any()
    assert not _np(net.dW[-1])[n:].any()
    return mag


@pytest.mark.parametrize("direct_first,save", [(True, "recompute"), (False, "recompute"),
                                               (True, "fused"), (False, "fused")])
def test_csnn_step_small_matches_oracle(direct_first, save, cuda_device):
    """The step at T = 4, B = 8, with the first layer as a direct
    convolution or as im2col + tensor-core GEMM, recomputing the membrane in
    the BPTT or (fused) storing it and scanning in the GEMM epilogues."""
    w = SMALL
    inp = _exact_inputs(w)
    convs, Wfc, betas, fwd, res = _oracle(w, inp, stored=save == "fused")
    assert all(s.mean() > 0 for s in fwd["spk"]) and fwd["fc_spk"].mean() > 0
    net, X, labels = _run(w, inp, cuda_device, direct_first=direct_first, save=save)
    assert net.direct[0] == direct_first
    net.step(X, labels)
    torch.cuda.synchronize()
    for layer in net.layers + [net.out_layer]:
        assert layer.status() == 0
    _check_step(w, net, convs, Wfc, betas, fwd, res)


def test_csnn_training_step_update_matches_oracle(cuda_device):
    """One full step (with AdamW on weights and betas): the updated fp32
    weights and betas equal the oracle's AdamW applied to the oracle's
    gradients, except where a gradient is within its tolerance of zero (Adam's
    first step is lr * sign(g) there, so either sign is correct)."""
    w = SMALL
    inp = _exact_inputs(w, W.SEED_BASE + 31)
    convs, Wfc, betas, fwd, res = _oracle(w, inp)
    hp = dict(lr=1e-2, betas=(0.9, 0.999), eps=1e-8, weight_decay=0.05)
    net, X, labels = _run(w, inp, cuda_device, **hp)
    net.train_step(X, labels)
    torch.cuda.synchronize()
    mag = _magnitudes(w, convs, Wfc, betas, fwd, np.abs(res["grad_out"]))
    lr, (b1, b2), eps, wd = hp["lr"], hp["betas"], hp["eps"], hp["weight_decay"]

    def expect(p, g, gmag, decay):
        new, _, _ = O.adamw_step(p, g, np.zeros_like(p), np.zeros_like(p), lr, b1, b2, eps, decay, 1)
        tol_g = GRAD_RTOL * np.maximum(gmag, np.abs(g)) + 1e-12
        ambiguous = np.abs(g) <= tol_g
        return new, np.where(ambiguous, 2 * lr, 1e-6 * (np.abs(p) + lr))

    for l in range(len(convs)):
        new, tol = expect(convs[l], res["dW"][l], mag["dW"][l], wd)
        H.assert_close(f"W{l}", _np(net.conv_weight(l)), new, 0.0, tol)
        new, tol = expect(betas[l], res["dbeta"][l], mag["dbeta"][l], 0.0)
        H.assert_close(f"beta{l}", _np(net.beta[l])[: len(betas[l])], new, 0.0, tol)
    new, tol = expect(Wfc, res["dW_fc"], mag["dW_fc"], wd)
    H.assert_close("Wfc", _np(net.fc_weight()), new, 0.0, tol)
    assert net.step_counter.cpu().tolist() == [1, 0]
    assert net.beta_counter.cpu().tolist() == [1, 0]
    assert torch.equal(net.W_flat.cpu(), net.W32_flat.cpu().to(torch.bfloat16))


@pytest.mark.parametrize("save", ["recompute", "fused"])
def test_csnn_step_full_size(save, cuda_device):
    """12C5-MP2-64C5-MP2-10 at T = 25, B = 128 (the configuration the
    benchmark times): the same exact forward and gradient bounds."""
    w = W.CSNN_C4
    inp = _exact_inputs(w)
    convs, Wfc, betas, fwd, res = _oracle(w, inp, stored=save == "fused")
    net, X, labels = _run(w, inp, cuda_device, save=save)
    net.step(X, labels)
    torch.cuda.synchronize()
    for layer in net.layers + [net.out_layer]:
        assert layer.status() == 0
    _check_step(w, net, convs, Wfc, betas, fwd, res)


def test_csnn_training_lowers_the_loss(cuda_device):
    w = W.CSNN_C4
    inp = W.make_conv_inputs(w)
    net, X, labels = _run(w, inp, cuda_device, lr=2e-3)
    losses = [float(net.train_step(X, labels).item())]
    for _ in range(29):
        losses.append(float(net.train_step(X, labels).item()))
    torch.cuda.synchronize()
    assert net.step_counter.cpu().tolist() == [30, 0]
    for layer in net.layers + [net.out_layer]:
        assert layer.status() == 0
    assert np.all(np.isfinite(losses))
    assert min(losses[-5:]) < 0.8 * losses[0], losses
    # the padded channels' betas never move
    for l, (c, _) in enumerate(w.convs):
        assert torch.all(net.beta[l][c:] == w.beta)


# ---------------------------------------------------------------------------
# Stage by stage with He-uniform weights as drawn (no flushing), teacher-forced
# ---------------------------------------------------------------------------

BF16_HALF_ULP = 2.0 ** -8   # |bf16 rounding error| <= 2^-8 |value|
ACC_RTOL = 1e-5             # fp32 accumulation, of the magnitude of the summed terms
GEMM_RTOL = 1e-5


def _close_bf16(name, got, ref, scale):
    """One bf16 rounding of an fp32 result: |got - ref| <= 2^-8 |ref| +
    1e-5 * scale (the magnitude of the summed terms); returns the count
    needing the scale term."""
    return H.assert_close(name, got, ref, BF16_HALF_ULP, ACC_RTOL * scale + 1e-30)


def _col2im(dcols, Hh, Ww, k):
    """Sum of the patch-row gradients [M, Ho, Wo, k, k, C] into the input
    map [M, Hh, Ww, C] (float64)."""
    M, Ho, Wo, _, _, C = dcols.shape
    out = np.zeros((M, Hh, Ww, C))
    for ky in range(k):
        for kx in range(k):
            out[:, ky:ky + Ho, kx:kx + Wo, :] += dcols[:, :, :, ky, kx, :]
    return out


def _scan_forced(w, l_name, I32, beta, zg, bound, counts, sizes, mem_gpu=None):
    """The oracle's float32 Leaky scan (Eq. 4, reset to zero) with its reset
    held at the GPU's spikes zg [T, L]; a GPU spike may differ from the
    oracle's decision only within the currents' error bound of the
    threshold.  Returns the trace the GPU's reverse pass reads (its stored
    bf16 trace, checked against the oracle's, or the oracle's fp32 one)."""
    T, L = zg.shape
    z_reset = np.vstack([np.zeros((1, L)), zg[:-1]])
    spk32, mem32 = O.leaky_forward(I32, beta.astype(np.float32), np.full(L, w.thr, np.float32),
                                   w.reset, dtype=np.float32, z_reset=z_reset)
    spk32, mem32 = spk32.astype(np.float64), mem32.astype(np.float64)
    diff = spk32 != zg
    allowed = np.maximum(H.AMBIGUITY, 2.0 * bound)
    assert np.all(np.abs(mem32 - w.thr)[diff] < allowed[diff]), f"{l_name}: spike off threshold"
    counts[f"{l_name}_spk_forced"], sizes[f"{l_name}_spk_forced"] = int(diff.sum()), T * L
    if mem_gpu is None:
        return mem32
    # the GPU rounds its own fp32 membrane, within 2 * bound of the oracle's:
    # rounding is monotone, so the stored value lies between the roundings
    # of the interval's ends
    exact = O.bf16_round(mem32)
    lo = O.bf16_round(mem32 - 2.0 * bound - 1e-7)
    hi = O.bf16_round(mem32 + 2.0 * bound + 1e-7)
    bad = ~((mem_gpu == exact) | ((mem_gpu >= lo) & (mem_gpu <= hi)))
    if bad.any():
        i = np.argwhere(bad)[:5]
        d = np.abs(mem_gpu - mem32)[bad]
        raise AssertionError(
            f"{l_name}: stored membrane: {bad.sum()} of {bad.size}; first {i.tolist()}; "
            f"gpu {mem_gpu[bad][:5]} oracle {mem32[bad][:5]} bound {bound[bad][:5]}; "
            f"max |diff| {d.max()}; forced here {diff[bad].sum()}")
    counts[f"{l_name}_mem_midpoint"] = int((mem_gpu != exact).sum())
    sizes[f"{l_name}_mem_midpoint"] = T * L
    return mem_gpu


def _bound(w, S, T, beta):
    """Running bound on the membrane from currents within GEMM_RTOL of their
    summed terms S [T, L] (Eq. 4 carries it with factor beta)."""
    e, out = np.zeros(S.shape[1]), np.zeros_like(S)
    for t in range(T):
        e = beta * e + GEMM_RTOL * S[t] + 1e-6 + 4 * H.EPS32 * (1.0 + S[t])
        out[t] = e
    return out


def check_csnn_stagewise(w, inp, net, widened_frac=1e-3):
    """Each stage of the CSNN step against the oracle's, fed the GPU's own
    inputs to that stage (teacher forcing at every element where several
    results are correct; see check_dsnn_stagewise).  Layout stages (pooling,
    its backward) must be exact functions of the GPU's inputs; every bf16
    result is one rounding of an fp32 one (2^-8 of |ref| plus 1e-5 of the
    summed terms); fp32 weight and beta gradients are within 1e-5 of their
    summed terms."""
    T, B, M = w.T, w.B, w.T * w.B
    convs = [_np(c) for c in inp["convs"]]
    Wfc = _np(inp["Wfc"])
    X = _np(inp["X"]).reshape(M, w.H, w.W, w.Cin)
    labels = _np(inp["labels"]).astype(np.int64)
    nl = len(convs)
    counts, sizes = {}, {}
    stored = net.layers[0].mem is not None
    ins, traces, spks = [], [], []
    x = X
    for l in range(nl):
        cout, k = w.convs[l]
        _, _, cin_p, cp, _, Ho, Wo, *_r = net.geo[l]
        L = B * Ho * Wo * cout
        I64 = O.conv2d_nhwc(x, convs[l])
        S = O.conv2d_nhwc(np.abs(x), np.abs(convs[l]))
        beta = np.tile(np.full(cout, w.beta), B * Ho * Wo)
        zg = _np(net.layers[l].spk).reshape(M, Ho, Wo, cp)[..., :cout].reshape(T, L)
        if net.I[l] is not None:
            Ig = _np(net.I[l]).reshape(M, Ho, Wo, cp)
            H.assert_close(f"I{l}", Ig[..., :cout], I64, GEMM_RTOL, 1e-6, S)
            I32, bound = Ig[..., :cout].reshape(T, L).astype(np.float32), np.zeros((T, L))
        else:
            I32 = I64.reshape(T, L).astype(np.float32)
            bound = _bound(w, S.reshape(T, L), T, w.beta)
        mem_g = None
        if stored:
            mem_g = _np(net.layers[l].mem).reshape(M, Ho, Wo, cp)[..., :cout].reshape(T, L)
        traces.append(_scan_forced(w, f"conv{l}", I32, beta, zg, bound, counts, sizes, mem_g))
        spks.append(zg)
        s = zg.reshape(M, Ho, Wo, cout)
        p, idx = O.maxpool2_nhwc(s)
        pg = _np(net.pool[l])
        assert np.array_equal(pg[..., :cout], p) and not pg[..., cout:].any(), f"pool {l}"
        assert np.array_equal(net.idx[l].cpu().numpy().astype(np.int64)[..., :cout], idx)
        ins.append(x)
        x = p
    n = w.n_classes
    flat = x.reshape(M, -1)
    Lf = B * n
    Ifc64 = O.dense_forward(flat, Wfc)
    Sfc = np.abs(flat) @ np.abs(Wfc).T
    zo = _np(net.out_layer.spk)[:, :, :n].reshape(T, Lf)
    if net.I_fc is not None:
        Ig = _np(net.I_fc)[:, :n]
        H.assert_close("I_fc", Ig, Ifc64, GEMM_RTOL, 1e-6, Sfc)
        I32, bound = Ig.reshape(T, Lf).astype(np.float32), np.zeros((T, Lf))
    else:
        I32, bound = Ifc64.reshape(T, Lf).astype(np.float32), _bound(w, Sfc.reshape(T, Lf), T,
                                                                      w.beta_fc)
    mem_o = _np(net.out_layer.mem)[:, :, :n].reshape(T, Lf) if stored else None
    trace_o = _scan_forced(w, "out", I32, np.full(Lf, w.beta_fc), zo, bound, counts, sizes, mem_o)

    # loss and readout
    loss_o, g_o = O.rate_ce_loss(zo.reshape(T, B, n), labels)
    assert abs(float(net.loss.item()) - loss_o) <= 1e-6 * max(1.0, abs(loss_o))
    go = _np(net.grad_out)
    H.assert_close("grad_out", go[:, :, :n], g_o, BF16_HALF_ULP, 1e-7)
    gs = g_o.reshape(T, Lf) if net.fused_loss else go[:, :, :n].reshape(T, Lf)
    kw = dict(reset=w.reset, detach=True, sg="fast_sigmoid", sg_param=w.sg_param)
    thr_o = np.full(Lf, w.thr)
    ref = O.leaky_backward(trace_o, zo, gs, np.full(Lf, w.beta_fc), thr_o, **kw)
    mag = O.leaky_backward(trace_o, zo, np.abs(gs), np.full(Lf, w.beta_fc), thr_o, **kw)
    gI = _np(net.out_layer.grad_I)[:, :, :n].reshape(T, Lf)
    counts["grad_I_fc"] = _close_bf16("grad_I_fc", gI, ref["grad_I"],
                                      np.maximum(mag["grad_I"], np.abs(ref["grad_I"])))
    sizes["grad_I_fc"] = T * Lf
    dI = gI.reshape(M, n)
    H.assert_close("dW_fc", _np(net.fc_weight(net.dW_flat)), dI.T @ flat, ACC_RTOL, 1e-12,
                   np.abs(dI).T @ np.abs(flat))
    d_flat, d_mag = dI @ Wfc, np.abs(dI) @ np.abs(Wfc)
    cl = w.convs[-1][0]
    gp = _np(net.grad_pool[-1])
    Hp, Wp, cpl = gp.shape[1], gp.shape[2], gp.shape[3]
    counts["grad_pool_top"] = _close_bf16("grad_pool_top", gp[..., :cl].reshape(M, -1), d_flat,
                                          d_mag)
    sizes["grad_pool_top"] = d_flat.size
    # the conv layers, top down
    for l in range(nl - 1, -1, -1):
        cout, k = w.convs[l]
        _, _, cin_p, cp, _, Ho, Wo, *_r = net.geo[l]
        L = B * Ho * Wo * cout
        gpool = _np(net.grad_pool[l])[..., :cout]
        _, idx = O.maxpool2_nhwc(spks[l].reshape(M, Ho, Wo, cout))
        d_spk = O.maxpool2_nhwc_backward(gpool, idx, (M, Ho, Wo, cout))
        gsp = _np(net.grad_spk[l]).reshape(M, Ho, Wo, cp)
        assert np.array_equal(gsp[..., :cout], d_spk) and not gsp[..., cout:].any(), \
            f"pool {l} backward"
        g = d_spk.reshape(T, L)
        beta = np.tile(np.full(cout, w.beta), B * Ho * Wo)
        ref = O.leaky_backward(traces[l], spks[l], g, beta, np.full(L, w.thr), **kw)
        mag = O.leaky_backward(traces[l], spks[l], np.abs(g), beta, np.full(L, w.thr), **kw)
        gI = _np(net.layers[l].grad_I).reshape(M, Ho, Wo, cp)
        counts[f"grad_I{l}"] = _close_bf16(f"grad_I{l}", gI[..., :cout].reshape(T, L),
                                           ref["grad_I"],
                                           np.maximum(mag["grad_I"], np.abs(ref["grad_I"])))
        sizes[f"grad_I{l}"] = T * L
        # per-channel beta: du_t * (1 - z_{t-1}) u_{t-1}, summed over t and the channel's lanes
        prev = np.vstack([np.zeros((1, L)), np.abs(traces[l][:-1])])
        db_mag = (mag["grad_I"] * prev).reshape(-1, cout).sum(axis=0)
        db_ref = O.reduce_lane_grad(ref["grad_beta_lane"], B, Ho * Wo * cout, "per_channel",
                                    C=cout, HW=1)
        H.assert_close(f"dbeta{l}", _np(net.dbeta[l])[:cout], db_ref, ACC_RTOL, 1e-9, db_mag)
        dIl = gI[..., :cout]
        dX, dW = O.conv2d_nhwc_backward(ins[l], convs[l], dIl)
        _, dW_mag = O.conv2d_nhwc_backward(np.abs(ins[l]), np.abs(convs[l]), np.abs(dIl))
        H.assert_close(f"dW{l}", _np(net.conv_weight(l, net.dW_flat)), dW, ACC_RTOL, 1e-12, dW_mag)
        if l > 0:
            # patch-row gradients (one rounding each), then col2im of the GPU's
            # patch rows (one rounding of their fp32 sum)
            cin = w.convs[l - 1][0]
            dc = _np(net.dcols[l])[:, : k * k * cin_p].reshape(M, Ho, Wo, k, k, cin_p)[..., :cin]
            W2 = convs[l].reshape(cout, -1)
            rows = dIl.reshape(-1, cout)
            dc_ref = (rows @ W2).reshape(M, Ho, Wo, k, k, cin)
            dc_mag = (np.abs(rows) @ np.abs(W2)).reshape(M, Ho, Wo, k, k, cin)
            counts[f"dcols{l}"] = _close_bf16(f"dcols{l}", dc, dc_ref, dc_mag)
            sizes[f"dcols{l}"] = dc.size
            Hh, Ww = ins[l].shape[1], ins[l].shape[2]
            gp = _np(net.grad_pool[l - 1])[..., :cin]
            ci_ref, ci_mag = _col2im(dc, Hh, Ww, k), _col2im(np.abs(dc), Hh, Ww, k)
            counts[f"col2im{l}"] = _close_bf16(f"col2im{l}", gp, ci_ref, ci_mag)
            sizes[f"col2im{l}"] = gp.size
    H.assert_widened(counts, sizes, widened_frac)
    return counts


@pytest.mark.parametrize("save", ["recompute", "fused"])
@pytest.mark.parametrize("w", [SMALL, W.CSNN_C4], ids=lambda w: w.name)
def test_csnn_step_real_weights_stagewise(w, save, cuda_device):
    """The step with the He-uniform weights as drawn (every sum rounds in
    fp32), at T = 4, B = 8 and at the benchmark's T = 25, B = 128: every
    element of every stage, teacher-forced."""
    inp = W.make_conv_inputs(w)
    net, X, labels = _run(w, inp, cuda_device, save=save)
    net.step(X, labels)
    torch.cuda.synchronize()
    for layer in net.layers + [net.out_layer]:
        assert layer.status() == 0
    print(w.name, save, check_csnn_stagewise(w, inp, net))
