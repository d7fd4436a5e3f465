"""Parity of the 3-layer dense SNN training step (Tab. I DSNN: dense GEMM ->
Leaky scan per layer, rate-coded CE loss, BPTT through all layers) with the
oracle's composition of the same steps.

Comparison protocol
-------------------
* Input currents: the GEMM sums bf16 products in fp32; it must agree with the
  float64 product within 1e-5 of the magnitude of the summed terms.  That
  bound, carried through Eq. (4) (e_t = beta e_{t-1} + e_I,t), bounds how far
  the kernel's membrane can sit from the oracle's float32 trace.
* Spikes are compared bit for bit.  At the small size the inputs are drawn
  (oracle only) until every decision of every layer is at least 1e-4 from
  the threshold, far beyond the fp32 rounding differences of the two sums
  (about 1e-6), so one spike train is expected.  At the full size a sample
  whose spikes differ anywhere is excluded from the later per-sample
  comparisons, and each such difference must sit where the oracle's membrane
  is within twice that bound of the threshold.
* With the bf16 membrane trace stored (save="mem"), a value whose fp32
  membrane lies within 1e-4 of a bf16 rounding midpoint may be stored either
  way; the surrogate then takes one of two values.  The oracle carries that
  choice as an uncertainty through the reverse pass (absolute values, the
  surrogate difference times the spike gradient as a source term) and the
  tolerance adds it.
* Gradients: the path keeps the loss gradient, every dL/dI and every dL/din
  in bf16 and the oracle rounds at the same points.  A rounding that goes the
  other way changes a value by at most one bf16 ulp (2^-7 of it); there are
  at most six such points between the loss and the deepest gradient, so the
  tolerance is 6 * 2^-7 of the magnitude of the summed terms (the reverse
  pass run on absolute values).
"""
import numpy as np
import pytest
import torch

from oracle import snn_oracle as O
from paper_2211_10725_gb300 import workloads as W
from paper_2211_10725_gb300.dsnn import DenseSNN
from tests import scan_harness as H

pytestmark = pytest.mark.gpu

GEMM_RTOL, GEMM_ATOL = 1e-5, 1e-6
GRAD_RTOL = 6 * 2.0 ** -7
MARGIN = 1e-4   # spike decisions / bf16 midpoints closer than this may differ

SMALL = W.DSNN_C3.scaled(name="dsnn_784_128_64_10_T6_B16", T=6, B=16, sizes=(784, 128, 64, 10))
SMALL_POP = W.DSNN_POP.scaled(name="dsnn_pop_784_128_60_T2_B16", T=2, B=16, sizes=(784, 128, 60),
                              pop=6)


def _np(t):
    return t.detach().to("cpu", torch.float32).numpy().astype(np.float64)


def _oracle(w, inp):
    Ws = [_np(x) for x in inp["W"]]
    X = _np(inp["X"]).reshape(w.T * w.B, -1)
    fwd = O.dsnn_forward(X, Ws, w.T, w.B, w.beta, w.thr, dtype=np.float32)
    return Ws, X, fwd


def _membrane_bounds(w, Ws, fwd):
    """Per layer [T, B*N] bound on |u_kernel - u_oracle| from the GEMM
    tolerance (same spike path assumed), plus float32 rounding of Eq. (4)."""
    out = []
    for l, Wl in enumerate(Ws):
        S = (np.abs(fwd["ins"][l]) @ np.abs(Wl).T).reshape(w.T, -1)
        e, bound = np.zeros(S.shape[1]), np.zeros_like(S)
        for t in range(w.T):
            e = w.beta * e + GEMM_RTOL * S[t] + GEMM_ATOL + 4 * H.EPS32 * (1.0 + S[t])
            bound[t] = e
        out.append(bound)
    return out


def _abs_reverse(w, Ws, fwd, g_top, sources=None):
    """The step's reverse pass on absolute values (every coefficient is then
    >= 0), from spike gradient g_top [T, B*C] of the last layer; sources[l]
    [T, B*N_l], if given, is added to dL/du of layer l at each step."""
    T, B = w.T, w.B
    gs = g_top
    out = {"grad_I": [None] * len(Ws), "dW": [None] * len(Ws)}
    for l in range(len(Ws) - 1, -1, -1):
        n = Ws[l].shape[0]
        g = O.leaky_backward(fwd["mem"][l], fwd["spk"][l], gs, np.full(B * n, w.beta),
                             np.full(B * n, w.thr), reset="subtract", detach=True,
                             sg="fast_sigmoid", sg_param=w.sg_param,
                             grad_mem=None if sources is None else sources[l])
        dI = g["grad_I"].reshape(T * B, n)
        dX, dW = O.dense_backward(np.abs(fwd["ins"][l]), np.abs(Ws[l]), dI)
        out["grad_I"][l], out["dW"][l] = dI, dW
        gs = dX.reshape(T, -1)
    return out


def _magnitudes(w, Ws, fwd, res):
    """For each gradient the magnitude of the terms it sums."""
    return _abs_reverse(w, Ws, fwd, np.abs(res["grad_out"]).reshape(w.T, -1))


def _storage_choice(w, mem32):
    """bf16 candidates of the stored trace: (lo, hi) differ where the fp32
    value is within MARGIN of a rounding midpoint."""
    return O.bf16_round(mem32 - MARGIN), O.bf16_round(mem32 + MARGIN)


def _storage_uncertainty(w, Ws, fwd32, res, mag):
    """Bound on how far the gradients move when the stored bf16 trace takes
    the other rounding where both are correct: the surrogate difference times
    the (magnitude of the) spike gradient at each such element, carried
    through the reverse pass on absolute values."""
    sources = []
    for l in range(len(Ws)):
        lo, hi = _storage_choice(w, fwd32["mem"][l])
        ds = np.abs(O.surrogate_grad(lo - w.thr, "fast_sigmoid", w.sg_param)
                    - O.surrogate_grad(hi - w.thr, "fast_sigmoid", w.sg_param))
        sources.append(ds * np.abs(res["grad_spk"][l]) * (1.0 + GRAD_RTOL))
    zero = np.zeros_like(res["grad_out"]).reshape(w.T, -1)
    return _abs_reverse(w, Ws, fwd32, zero, sources)


def _run(w, inp, device, save="recompute"):
    net = DenseSNN(w, inp["W"], device=device, save=save)
    X = inp["X"].reshape(w.T * w.B, -1).to(device)
    labels = inp["labels"].to(device)
    net.step(X, labels)
    torch.cuda.synchronize()
    for layer in net.layers:
        assert layer.status() == 0
    return net


def _gpu_layer(net, l):
    """GPU results of layer l without the padding neurons."""
    w = net.w
    n, k = net.sizes[l + 1], net.sizes[l]
    layer = net.layers[l]
    return {
        "I": None if net.I[l] is None else _np(net.I[l])[:, :n],
        "spk": _np(layer.spk)[:, :, :n],
        "grad_I": _np(layer.grad_I)[:, :, :n].reshape(w.T * w.B, n),
        "dW": _np(net.dW[l])[:n, :k],
        "pad": (_np(layer.spk)[:, :, n:], _np(layer.grad_I)[:, :, n:], _np(net.dW[l])[n:, :],
                _np(net.dW[l])[:, k:]),
    }


def _small_seed(w):
    """First seed whose oracle run has every spike decision of every layer
    at least MARGIN from the threshold, with every layer spiking."""
    for s in range(200):
        seed = W.SEED_BASE + 1000 + s
        inp = W.make_dense_inputs(w, seed)
        Ws, X, fwd = _oracle(w, inp)
        ok = all(0.0 < f.mean() for f in fwd["spk"])
        ok = ok and all(bool(np.all(np.abs(m - w.thr) > MARGIN)) for m in fwd["mem"])
        if ok:
            return seed
    raise AssertionError("no seed with clear spike decisions")


@pytest.mark.parametrize("w,save", [(SMALL, "recompute"), (SMALL, "mem"), (SMALL, "fused"),
                                    (SMALL_POP, "recompute"), (SMALL_POP, "fused")])
def test_dsnn_step_small_matches_oracle(w, save, cuda_device):
    seed = _small_seed(w)
    inp = W.make_dense_inputs(w, seed)
    Ws, X, fwd = _oracle(w, inp)
    net = _run(w, inp, cuda_device, save)
    T, B = w.T, w.B
    store = O.bf16_round
    fwd32 = fwd
    stored = save in ("mem", "fused")  # the backward reads the stored bf16 trace
    if stored:
        # the backward reads the bf16 trace the forward stored
        fwd = dict(fwd, mem=[store(m) for m in fwd["mem"]])
    res = O.dsnn_backward(fwd, Ws, _np(inp["labels"]).astype(np.int64), T, B, w.beta, w.thr,
                          w.sg_param, store=store, pop=w.pop)
    mag = _magnitudes(w, Ws, fwd, res)
    unc = _storage_uncertainty(w, Ws, fwd32, res, mag) if stored else None

    loss = float(net.loss.item())
    assert abs(loss - res["loss"]) <= 1e-6 * max(1.0, abs(res["loss"]))
    go = _np(net.grad_out)
    C = w.sizes[-1]
    H.assert_close("grad_out", go[:, :, :C], res["grad_out"], 2.0 ** -7, 0.0)
    assert not go[:, :, C:].any()
    for l in range(len(Ws)):
        g = _gpu_layer(net, l)
        S = np.abs(fwd["ins"][l]) @ np.abs(Ws[l]).T
        if g["I"] is not None:  # the fused forward keeps its currents on chip
            H.assert_close(f"I{l}", g["I"], fwd["I"][l], GEMM_RTOL, GEMM_ATOL, S)
        assert np.array_equal(g["spk"].reshape(T, -1), fwd["spk"][l]), f"layer {l} spikes"
        extra_I, extra_W = 0.0, 0.0
        if stored:
            n = w.sizes[l + 1]
            got = _np(net.layers[l].mem)[:, :, :n].reshape(T, -1)
            lo, hi = _storage_choice(w, fwd32["mem"][l])
            assert np.all((got == fwd["mem"][l]) | (got == lo) | (got == hi)), \
                f"layer {l} stored membrane"
            extra_I, extra_W = unc["grad_I"][l], unc["dW"][l]
        H.assert_close(f"grad_I{l}", g["grad_I"], res["grad_I"][l], GRAD_RTOL, 1e-12 + extra_I,
                       np.maximum(mag["grad_I"][l], np.abs(res["grad_I"][l])))
        H.assert_close(f"dW{l}", g["dW"], res["dW"][l], GRAD_RTOL, 1e-12 + extra_W,
                       np.maximum(mag["dW"][l], np.abs(res["dW"][l])))
        for p in g["pad"]:
            assert not p.any(), f"layer {l} padding not zero"


@pytest.mark.parametrize("save", ["recompute", "fused"])
@pytest.mark.parametrize("w", [W.DSNN_C3, W.DSNN_POP], ids=lambda w: w.name)
def test_dsnn_step_full_size(w, save, cuda_device):
    """784-1000-1000-10, T = 25, B = 128, and the population-coded
    3072-1000-500 network at T = 1 (the configurations timed by the
    benchmark, which uses the fused forward): per-sample parity for every
    sample whose spikes match in all layers, ambiguity-only differences
    elsewhere, and dW close overall.  With the stored bf16 trace the
    gradients may also move by the storage uncertainty."""
    inp = W.make_dense_inputs(w)
    Ws, X, fwd = _oracle(w, inp)
    net = _run(w, inp, cuda_device, save)
    fwd32 = fwd
    T, B = w.T, w.B
    bounds = _membrane_bounds(w, Ws, fwd)
    clean = np.ones(B, dtype=bool)
    for l in range(len(Ws)):
        g = _gpu_layer(net, l)
        n = w.sizes[l + 1]
        S = (np.abs(fwd["ins"][l]) @ np.abs(Ws[l]).T).reshape(T, B, n)
        if g["I"] is not None:  # the fused forward keeps its currents on chip
            Ig = g["I"].reshape(T, B, n)[:, clean]
            H.assert_close(f"I{l}", Ig, fwd["I"][l].reshape(T, B, n)[:, clean], GEMM_RTOL,
                           GEMM_ATOL, S[:, clean])
        so = fwd["spk"][l].reshape(T, B, n)
        diff = (g["spk"] != so) & clean[None, :, None]
        margin = np.abs(fwd["mem"][l].reshape(T, B, n) - w.thr)
        allowed = np.maximum(MARGIN, 2.0 * bounds[l].reshape(T, B, n))
        assert np.all(margin[diff] < allowed[diff]), \
            f"layer {l}: spike difference away from the threshold"
        clean &= ~diff.any(axis=(0, 2))
        assert not g["pad"][0].any()
    assert clean.sum() >= B // 2, f"only {clean.sum()} samples agree in every layer"

    if save == "fused":
        fwd = dict(fwd, mem=[O.bf16_round(m) for m in fwd["mem"]])
    res = O.dsnn_backward(fwd, Ws, _np(inp["labels"]).astype(np.int64), T, B, w.beta, w.thr,
                          w.sg_param, store=O.bf16_round, pop=w.pop)
    mag = _magnitudes(w, Ws, fwd, res)
    unc = _storage_uncertainty(w, Ws, fwd32, res, mag) if save == "fused" else None
    for l in range(len(Ws)):
        g = _gpu_layer(net, l)
        n = w.sizes[l + 1]
        gi = g["grad_I"].reshape(T, B, n)[:, clean]
        ri = res["grad_I"][l].reshape(T, B, n)[:, clean]
        sc = np.maximum(mag["grad_I"][l].reshape(T, B, n)[:, clean], np.abs(ri))
        extra = 0.0 if unc is None else unc["grad_I"][l].reshape(T, B, n)[:, clean]
        H.assert_close(f"grad_I{l}", gi, ri, GRAD_RTOL, 1e-12 + extra, sc)
        # dW sums over all samples, including any that took another spike path
        rel = np.linalg.norm(g["dW"] - res["dW"][l]) / np.linalg.norm(res["dW"][l])
        allowed = GRAD_RTOL + 2.0 * (B - clean.sum()) / B
        if unc is not None:
            allowed += np.linalg.norm(unc["dW"][l]) / np.linalg.norm(res["dW"][l])
        assert rel < allowed, f"dW{l} relative error {rel:.3g} (allowed {allowed:.3g})"
    if clean.all():
        assert abs(float(net.loss.item()) - res["loss"]) <= 1e-6 * max(1.0, abs(res["loss"]))
