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


# ---------------------------------------------------------------------------
# Stage-by-stage comparison, teacher-forced (every sample, any seed)
# ---------------------------------------------------------------------------

BF16_HALF_ULP = 2.0 ** -8   # |bf16 rounding error| <= 2^-8 |value|
ACC_RTOL = 1e-5             # fp32 accumulation, of the magnitude of the summed terms


def check_dsnn_stagewise(w, inp, net, save, widened_frac=1e-3):
    """Each stage of the step against the oracle's, fed the GPU's own inputs
    to that stage (the comparison protocol: the oracle follows the GPU at
    every element where several results are correct, so every sample stays
    on one path and everything is compared).

    Forward, per layer: the layer's input is the GPU's spikes of the layer
    below; the float64 GEMM bounds the GPU's currents; the oracle's float32
    Leaky scan runs with its reset held at the GPU's spikes, and a GPU spike
    may differ from the oracle's decision only where the oracle's membrane
    is within the currents' error bound (carried through Eq. 4) of the
    threshold; the stored bf16 trace must be the rounding of the oracle's
    membrane or, within that bound of a rounding midpoint, its neighbour.
    Backward, per layer from the top: the oracle's BPTT runs on the trace and
    spikes the GPU's reverse pass reads and on the spike gradient the GPU
    formed (the loss gradient; the GPU's bf16 dL/dspk where it is stored;
    else the float64 product of the GPU's dL/dI of the layer above with W).
    Every dL/dI is one bf16 rounding of an fp32 result: |gpu - ref| <=
    2^-8 |ref| + 1e-5 * (magnitude of the summed terms).  dW is the fp32
    product of the GPU's dL/dI and the layer input: 1e-5 of its terms.
    Returns the counts of forced spikes and of elements judged by the
    summed-terms band; each is bounded by `widened_frac` of its output."""
    T, B = w.T, w.B
    Ws = [_np(x) for x in inp["W"]]
    X = _np(inp["X"]).reshape(T * B, -1)
    labels = _np(inp["labels"]).astype(np.int64)
    nl = len(Ws)
    gpu = [_gpu_layer(net, l) for l in range(nl)]
    stored = save in ("mem", "fused")
    counts, sizes = {}, {}
    ins = [X] + [gpu[l]["spk"].reshape(T * B, -1) for l in range(nl - 1)]
    traces = []
    for l in range(nl):
        n = w.sizes[l + 1]
        L = B * n
        S = np.abs(ins[l]) @ np.abs(Ws[l]).T                     # [T*B, n] summed terms
        I64 = O.dense_forward(ins[l], Ws[l])
        zg = gpu[l]["spk"].reshape(T, L)
        z_reset = np.vstack([np.zeros((1, L)), zg[:-1]])
        beta32, thr32 = np.full(L, w.beta, np.float32), np.full(L, w.thr, np.float32)
        if gpu[l]["I"] is not None:
            # the currents are materialised: check them, then take them as the
            # scan's input, so the oracle's float32 trace is the one the GPU
            # computes (and recomputes in the reverse pass)
            H.assert_close(f"I{l}", gpu[l]["I"], I64, GEMM_RTOL, GEMM_ATOL, S)
            I32 = gpu[l]["I"].astype(np.float32).reshape(T, L)
            bound = np.full((T, L), 0.0)
        else:
            I32 = I64.astype(np.float32).reshape(T, L)
            e, bound = np.zeros(L), np.zeros((T, L))
            for t in range(T):
                Sr = S.reshape(T, L)[t]
                e = w.beta * e + GEMM_RTOL * Sr + GEMM_ATOL + 4 * H.EPS32 * (1.0 + Sr)
                bound[t] = e
        spk32, mem32 = O.leaky_forward(I32, beta32, thr32, "subtract", dtype=np.float32,
                                       z_reset=z_reset)
        spk32, mem32 = spk32.astype(np.float64), mem32.astype(np.float64)
        diff = spk32 != zg
        allowed = np.maximum(H.AMBIGUITY, 2.0 * bound)
        margin = np.abs(mem32 - w.thr)
        assert np.all(margin[diff] < allowed[diff]), f"layer {l}: spike away from the threshold"
        counts[f"spk{l}_forced"], sizes[f"spk{l}_forced"] = int(diff.sum()), T * L
        if stored:
            got = _np(net.layers[l].mem)[:, :, :n].reshape(T, L)
            # the GPU rounds its own fp32 membrane, within 2 * bound of the
            # oracle's: rounding is monotone, so the stored value lies between
            # the roundings of the interval's ends
            exact = O.bf16_round(mem32)
            lo = O.bf16_round(mem32 - 2.0 * bound - 1e-7)
            hi = O.bf16_round(mem32 + 2.0 * bound + 1e-7)
            assert np.all((got == exact) | ((got >= lo) & (got <= hi))), \
                f"layer {l}: stored membrane"
            counts[f"mem{l}_midpoint"], sizes[f"mem{l}_midpoint"] = int((got != exact).sum()), T * L
            traces.append(got)
        else:
            traces.append(mem32)

    # the loss on the GPU's output spikes
    C = w.sizes[-1]
    loss_o, g_o = O.rate_ce_loss(gpu[-1]["spk"], labels, w.pop)
    assert abs(float(net.loss.item()) - loss_o) <= 1e-6 * max(1.0, abs(loss_o))
    go = _np(net.grad_out)
    H.assert_close("grad_out", go[:, :, :C], g_o, BF16_HALF_ULP, 1e-7)
    assert not go[:, :, C:].any()

    # the reverse pass, top down
    dI_up = None
    for l in range(nl - 1, -1, -1):
        n, k = w.sizes[l + 1], w.sizes[l]
        L = B * n
        if l == nl - 1:
            # with the readout's trace stored, the loss launch runs the
            # readout's BPTT on its fp32 class gradient; else the reverse
            # scan reads the stored bf16 loss gradient
            gs = g_o.reshape(T, L) if net.fused_loss else go[:, :, :C].reshape(T, L)
            gs_mag = np.abs(gs)
        else:
            dX = (dI_up @ Ws[l + 1]).reshape(T, L)
            dX_mag = (np.abs(dI_up) @ np.abs(Ws[l + 1])).reshape(T, L)
            if net.fused_bwd:
                gs, gs_mag = dX, dX_mag     # kept in fp32 on chip
            else:
                gin = _np(net.grad_in[l])[:, :n].reshape(T, L)
                counts[f"grad_spk{l}"] = _close_bf16(f"grad_spk{l}", gin, dX, dX_mag)
                sizes[f"grad_spk{l}"] = T * L
                gs, gs_mag = gin, np.abs(gin)
        kw = dict(reset="subtract", detach=True, sg="fast_sigmoid", sg_param=w.sg_param)
        beta, thr = np.full(L, w.beta), np.full(L, w.thr)
        ref = O.leaky_backward(traces[l], gpu[l]["spk"].reshape(T, L), gs, beta, thr, **kw)
        mag = O.leaky_backward(traces[l], gpu[l]["spk"].reshape(T, L), gs_mag, beta, thr, **kw)
        got = gpu[l]["grad_I"].reshape(T, L)
        counts[f"grad_I{l}"] = _close_bf16(f"grad_I{l}", got, ref["grad_I"],
                                           np.maximum(mag["grad_I"], np.abs(ref["grad_I"])))
        sizes[f"grad_I{l}"] = T * L
        dI = got.reshape(T * B, n)
        dW_ref = dI.T @ ins[l]
        dW_mag = np.abs(dI).T @ np.abs(ins[l])
        H.assert_close(f"dW{l}", gpu[l]["dW"], dW_ref, ACC_RTOL, 1e-12, dW_mag)
        for p_ in gpu[l]["pad"]:
            assert not p_.any(), f"layer {l} padding not zero"
        dI_up = dI
    H.assert_widened(counts, sizes, widened_frac)
    return counts


def _close_bf16(name, got, ref, scale):
    """One bf16 rounding of an fp32 result: |got - ref| <= 2^-8 |ref| +
    1e-5 * scale; returns the count needing the scale term."""
    return H.assert_close(name, got, ref, BF16_HALF_ULP, ACC_RTOL * scale + 1e-30)


@pytest.mark.parametrize("save", ["recompute", "mem", "fused"])
@pytest.mark.parametrize("w", [W.DSNN_C3, W.DSNN_POP], ids=lambda w: w.name)
def test_dsnn_step_full_size_stagewise(w, save, cuda_device):
    """784-1000-1000-10, T = 25, B = 128, and the population-coded
    3072-1000-500 network at T = 1 (the configurations the benchmark times,
    which uses save="fused"): every sample and every element, stage by
    stage, teacher-forced where several results are correct."""
    inp = W.make_dense_inputs(w)
    net = _run(w, inp, cuda_device, save)
    counts = check_dsnn_stagewise(w, inp, net, save)
    print(w.name, save, counts)


@pytest.mark.parametrize("save", ["recompute", "fused"])
def test_dsnn_step_small_unfiltered_seed_stagewise(save, cuda_device):
    """The small network on its workload's own seed (no search for clear
    spike decisions), stage by stage."""
    inp = W.make_dense_inputs(SMALL)
    net = _run(SMALL, inp, cuda_device, save)
    check_dsnn_stagewise(SMALL, inp, net, save)
