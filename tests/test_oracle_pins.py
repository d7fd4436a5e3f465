"""Pins for the CPU oracle: each test checks it against something the paper or
the mathematics fixes, not against a retyped copy of its own formulas.

* hand-worked traces of Eqs. (3)-(6) (exact values worked out by hand),
* closed forms of the spike-free linear recurrences,
* brute force: the unique self-consistent spike pattern of Eq. (3),
* BPTT against central finite differences of a smooth forward whose exact
  derivative is the surrogate (Sec. III-B, Eqs. 8-9),
* library routines (bfloat16 rounding, matmul, log-softmax autograd).
"""
import itertools
import math

import numpy as np
import pytest
import torch

from oracle import snn_oracle as O


# ---------------------------------------------------------------------------
# P4: hand-worked forward traces (values computed by hand from Eqs. 3-6)
# ---------------------------------------------------------------------------

I5 = np.array([0.5, 0.8, 0.3, 1.2, 0.0])[:, None]


@pytest.mark.parametrize("dtype,tol", [(np.float64, 1e-12), (np.float32, 2e-6)])
def test_hand_trace_leaky_subtract(dtype, tol):
    spk, mem = O.leaky_forward(I5, [0.9], [1.0], "subtract", dtype=dtype)
    assert spk[:, 0].tolist() == [0, 1, 0, 1, 0]
    np.testing.assert_allclose(mem[:, 0], [0.5, 1.25, 0.425, 1.5825, 0.42425], atol=tol)


@pytest.mark.parametrize("dtype,tol", [(np.float64, 1e-12), (np.float32, 2e-6)])
def test_hand_trace_leaky_zero_reset(dtype, tol):
    spk, mem = O.leaky_forward(I5, [0.9], [1.0], "zero", dtype=dtype)
    assert spk[:, 0].tolist() == [0, 1, 0, 1, 0]
    np.testing.assert_allclose(mem[:, 0], [0.5, 1.25, 0.3, 1.47, 0.0], atol=tol)


@pytest.mark.parametrize("dtype,tol", [(np.float64, 1e-12), (np.float32, 4e-6)])
def test_hand_trace_synaptic_subtract(dtype, tol):
    spk, mem, syn = O.synaptic_forward(I5, [0.8], [0.9], [1.0], "subtract", dtype=dtype)
    assert spk[:, 0].tolist() == [0, 1, 1, 1, 1]
    np.testing.assert_allclose(syn[:, 0], [0.5, 1.2, 1.26, 2.208, 1.7664], atol=tol)
    np.testing.assert_allclose(mem[:, 0], [0.5, 1.65, 1.745, 2.7785, 3.26705], atol=tol)


@pytest.mark.parametrize("dtype", [np.float64, np.float32])
def test_tie_at_threshold_does_not_fire(dtype):
    # Eq. (3) is strict: u == thr gives no spike.  0.5*0 + 1.0 == 1.0 exactly.
    spk, mem = O.leaky_forward(np.array([[1.0]]), [0.5], [1.0], dtype=dtype)
    assert mem[0, 0] == 1.0 and spk[0, 0] == 0.0


def test_reset_none_never_resets():
    spk, mem = O.leaky_forward(I5, [0.9], [1.0], "none")
    # without reset, u is the plain leaky sum even after spikes
    expect = [0.5, 1.25, 1.425, 2.4825, 2.23425]
    np.testing.assert_allclose(mem[:, 0], expect, atol=1e-12)
    assert spk[:, 0].tolist() == [0, 1, 1, 1, 1]


# ---------------------------------------------------------------------------
# P5: hand-worked BPTT, T=3 (values worked out by hand from the adjoint)
# ---------------------------------------------------------------------------

def _p5(detach):
    I = np.array([0.5, 0.8, 0.3])[:, None]
    spk, mem = O.leaky_forward(I, [0.9], [1.0], "subtract")
    return O.leaky_backward(mem, spk, np.ones((3, 1)), [0.9], [1.0], "subtract",
                            detach=detach, sg="fast_sigmoid", sg_param=1.0)


def test_hand_bptt_detached():
    g = _p5(True)
    np.testing.assert_allclose(g["grad_I"][:, 0], [1.346975057, 1.002811791, 0.403124213],
                               atol=2e-9)
    np.testing.assert_allclose(g["grad_beta_lane"][0], 1.005311162, atol=2e-9)
    np.testing.assert_allclose(g["grad_thr_lane"][0], -1.890692870, atol=2e-9)


def test_hand_bptt_not_detached():
    g = _p5(False)
    np.testing.assert_allclose(g["grad_I"][:, 0], [0.783747823, 0.744812295, 0.403124213],
                               atol=2e-9)
    np.testing.assert_allclose(g["grad_beta_lane"][0], 0.876311413, atol=2e-9)
    np.testing.assert_allclose(g["grad_thr_lane"][0], -1.301665687, atol=2e-9)


def test_fast_sigmoid_slope_one_is_eq9():
    # Eq. (9): 1/(1+|thr-u|)^2
    x = np.linspace(-3, 3, 61)
    np.testing.assert_allclose(O.surrogate_grad(x, "fast_sigmoid", 1.0),
                               1.0 / (1.0 + np.abs(-x)) ** 2, rtol=0, atol=0)


def test_atan_surrogate_integrates_to_one():
    # the arctan surrogate is a density: its integral over the real line is 1
    x = np.linspace(-2000, 2000, 4_000_001)
    val = np.trapezoid(O.surrogate_grad(x, "atan", 2.0), x)
    assert abs(val - 1.0) < 1e-3


# ---------------------------------------------------------------------------
# P1-P3: closed forms without spikes
# ---------------------------------------------------------------------------

def test_closed_form_leaky_no_spike():
    rng = np.random.default_rng(1)
    T, L = 40, 7
    I = rng.normal(0.2, 0.5, (T, L))
    beta = rng.uniform(0.5, 0.99, L)
    spk, mem = O.leaky_forward(I, beta, np.full(L, 1e30))
    assert spk.sum() == 0
    for t in range(T):
        expect = sum(beta ** (t - s) * I[s] for s in range(t + 1))
        np.testing.assert_allclose(mem[t], expect, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("equal", [False, True])
def test_closed_form_synaptic_no_spike(equal):
    rng = np.random.default_rng(2)
    T, L = 30, 5
    I = rng.normal(0.1, 0.4, (T, L))
    beta = rng.uniform(0.6, 0.95, L)
    alpha = beta.copy() if equal else rng.uniform(0.3, 0.55, L)
    spk, mem, syn = O.synaptic_forward(I, alpha, beta, np.full(L, 1e30))
    for t in range(T):
        isum = sum(alpha ** (t - s) * I[s] for s in range(t + 1))
        if equal:
            usum = sum(I[s] * (t - s + 1) * beta ** (t - s) for s in range(t + 1))
        else:
            usum = sum(I[s] * (beta ** (t - s + 1) - alpha ** (t - s + 1)) / (beta - alpha)
                       for s in range(t + 1))
        np.testing.assert_allclose(syn[t], isum, rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(mem[t], usum, rtol=1e-11, atol=1e-12)


def test_constant_input_steady_state():
    T = 400
    I = np.full((T, 3), 0.05)
    beta = np.array([0.9, 0.95, 0.5])
    _, mem = O.leaky_forward(I, beta, np.full(3, 1e30))
    ss = 0.05 / (1 - beta)
    for t in (0, 10, 100, T - 1):
        np.testing.assert_allclose(ss - mem[t], beta ** (t + 1) * ss, rtol=1e-9, atol=1e-13)
    alpha = np.array([0.8, 0.3, 0.6])
    _, mem, syn = O.synaptic_forward(I, alpha, beta, np.full(3, 1e30))
    np.testing.assert_allclose(syn[-1], 0.05 / (1 - alpha), rtol=1e-12)
    np.testing.assert_allclose(mem[-1], 0.05 / ((1 - alpha) * (1 - beta)), rtol=1e-7)


def test_closed_form_no_spike_gradients():
    # u_t = sum_s beta^(t-s) I_s  =>  dL/dI_s = sum_{t>=s} beta^(t-s) gm_t  and
    # dL/dbeta = sum_t gm_t sum_{s<t} (t-s) beta^(t-s-1) I_s   (sigma' ~ 0 far
    # from a threshold at 1e30 only through gm)
    rng = np.random.default_rng(3)
    T, L = 12, 4
    I = rng.normal(0.0, 1.0, (T, L))
    beta = rng.uniform(0.5, 0.95, L)
    gm = rng.normal(0.0, 1.0, (T, L))
    thr = np.full(L, 1e30)
    spk, mem = O.leaky_forward(I, beta, thr)
    g = O.leaky_backward(mem, spk, np.zeros((T, L)), beta, thr, grad_mem=gm)
    for s in range(T):
        np.testing.assert_allclose(
            g["grad_I"][s], sum(beta ** (t - s) * gm[t] for t in range(s, T)), rtol=1e-12)
    db = sum(gm[t] * sum((t - s) * beta ** (t - s - 1) * I[s] for s in range(t))
             for t in range(T))
    np.testing.assert_allclose(g["grad_beta_lane"], db, rtol=1e-10)


# ---------------------------------------------------------------------------
# P8: brute force — the spike train is the unique self-consistent pattern
# ---------------------------------------------------------------------------

def _consistent_patterns(I, beta, thr, reset):
    """Enumerate all z in {0,1}^T; for each, evaluate u from Eq. (4) with the
    pattern fixed, and keep the patterns with z_t == [u_t > thr] for all t."""
    T = len(I)
    keep = []
    for z in itertools.product((0, 1), repeat=T):
        u, ok, u_prev, z_prev = [], True, 0.0, 0
        for t in range(T):
            if reset == "subtract":
                ut = beta * u_prev + I[t] - z_prev * thr
            else:
                ut = beta * (1 - z_prev) * u_prev + I[t]
            if (ut > thr) != bool(z[t]):
                ok = False
                break
            u.append(ut)
            u_prev, z_prev = ut, z[t]
        if ok:
            keep.append((z, u))
    return keep


@pytest.mark.parametrize("reset", ["subtract", "zero"])
def test_brute_force_spike_patterns(reset):
    rng = np.random.default_rng(4)
    for trial in range(60):
        T = int(rng.integers(1, 6))
        I = rng.normal(0.6, 0.7, T)
        beta = float(rng.uniform(0.3, 0.99))
        pats = _consistent_patterns(I, beta, 1.0, reset)
        assert len(pats) == 1
        z, u = pats[0]
        spk, mem = O.leaky_forward(I[:, None], [beta], [1.0], reset)
        assert tuple(int(v) for v in spk[:, 0]) == z
        np.testing.assert_allclose(mem[:, 0], u, atol=1e-12)


# ---------------------------------------------------------------------------
# P6: BPTT equals the exact gradient of a smooth forward (central FD)
# ---------------------------------------------------------------------------

def _loss_smooth(neuron, p, gs, gm, gmf, gsf, reset, sg, k, z_reset):
    f = lambda x_thr: (lambda u: O.smooth_spike(u - x_thr, sg, k))
    if neuron == "leaky":
        spk, mem = O.leaky_forward(p["I"], p["beta"], p["thr"], reset, mem0=p["mem0"],
                                   spike_fn=f(p["thr"]), z_reset=z_reset)
        syn = None
    else:
        spk, mem, syn = O.synaptic_forward(p["I"], p["alpha"], p["beta"], p["thr"], reset,
                                           mem0=p["mem0"], syn0=p["syn0"],
                                           spike_fn=f(p["thr"]), z_reset=z_reset)
    L = (gs * spk).sum() + (gm * mem).sum() + (gmf * mem[-1]).sum()
    if syn is not None:
        L += (gsf * syn[-1]).sum()
    return L, spk, mem, syn


@pytest.mark.parametrize("neuron", ["leaky", "synaptic"])
@pytest.mark.parametrize("reset", ["subtract", "zero", "none"])
@pytest.mark.parametrize("detach", [True, False])
@pytest.mark.parametrize("sg,k", [("fast_sigmoid", 2.0), ("atan", 2.0)])
def test_bptt_matches_finite_differences(neuron, reset, detach, sg, k):
    rng = np.random.default_rng(hash((neuron, reset, detach, sg)) % 2**32)
    T, L = 5, 3
    p = {"I": rng.normal(0.6, 0.6, (T, L)), "beta": rng.uniform(0.5, 0.95, L),
         "thr": rng.uniform(0.7, 1.2, L), "mem0": rng.normal(0.5, 0.5, L),
         "alpha": rng.uniform(0.3, 0.9, L), "syn0": rng.normal(0.0, 0.3, L)}
    gs, gm = rng.normal(0, 1, (T, L)), rng.normal(0, 0.5, (T, L))
    gmf, gsf = rng.normal(0, 1, L), rng.normal(0, 1, L)
    L0, spk, mem, syn = _loss_smooth(neuron, p, gs, gm, gmf, gsf, reset, sg, k, None)
    z_init = O.smooth_spike(p["mem0"] - p["thr"], sg, k)
    # detached reset: the reset term's z_{t-1} is a constant held at its value
    z_reset = np.vstack([z_init[None], spk[:-1]]) if detach else None
    kw = dict(reset=reset, detach=detach, sg=sg, sg_param=k, grad_mem=gm,
              grad_mem_final=gmf, mem0=p["mem0"], z_init=z_init)
    if neuron == "leaky":
        g = O.leaky_backward(mem, spk, gs, p["beta"], p["thr"], **kw)
    else:
        g = O.synaptic_backward(mem, spk, syn, gs, p["alpha"], p["beta"], p["thr"],
                                syn0=p["syn0"], grad_syn_final=gsf, **kw)
    h = 1e-6

    def fd(name, idx):
        q = {kk: v.copy() for kk, v in p.items()}
        q[name][idx] += h
        lp = _loss_smooth(neuron, q, gs, gm, gmf, gsf, reset, sg, k, z_reset)[0]
        q[name][idx] -= 2 * h
        lm = _loss_smooth(neuron, q, gs, gm, gmf, gsf, reset, sg, k, z_reset)[0]
        return (lp - lm) / (2 * h)

    for t in range(T):
        for l in range(L):
            np.testing.assert_allclose(g["grad_I"][t, l], fd("I", (t, l)), rtol=1e-6, atol=1e-8)
    names = [("beta", "grad_beta_lane"), ("thr", "grad_thr_lane"), ("mem0", "grad_mem0")]
    if neuron == "synaptic":
        names += [("alpha", "grad_alpha_lane"), ("syn0", "grad_syn0")]
    # with a detached reset the FD holds the reset constants z_{t-1} fixed, so
    # the threshold's and mem0's effect through them is excluded on both sides
    for pname, gname in names:
        for l in range(L):
            np.testing.assert_allclose(g[gname][l], fd(pname, l), rtol=1e-6, atol=1e-8)


def test_surrogate_zero_limit_matches_hard_fd():
    # P7: with the true Heaviside and no membrane value near the threshold, a
    # small perturbation never flips a spike, so FD of the hard forward equals
    # BPTT with sigma' -> 0 (fast sigmoid with a huge slope).
    rng = np.random.default_rng(7)
    T, L = 8, 4
    I = rng.normal(0.5, 0.6, (T, L))
    beta, thr = np.full(L, 0.8), np.full(L, 1.0)
    gm = rng.normal(0, 1, (T, L))
    for reset in ("subtract", "zero"):
        spk, mem = O.leaky_forward(I, beta, thr, reset)
        assert np.abs(mem - 1.0).min() > 1e-3
        g = O.leaky_backward(mem, spk, np.zeros((T, L)), beta, thr, reset, detach=True,
                             sg="fast_sigmoid", sg_param=1e12, grad_mem=gm)
        h = 1e-7
        for t in range(T):
            Ip, Im = I.copy(), I.copy()
            Ip[t] += h
            Im[t] -= h
            fp = (gm * O.leaky_forward(Ip, beta, thr, reset)[1]).sum(axis=0)
            fm = (gm * O.leaky_forward(Im, beta, thr, reset)[1]).sum(axis=0)
            np.testing.assert_allclose(g["grad_I"][t], (fp - fm) / (2 * h), rtol=1e-6, atol=1e-9)


# ---------------------------------------------------------------------------
# Parameter layouts
# ---------------------------------------------------------------------------

def test_per_channel_mapping_isolates_one_channel():
    # Channel c of a [C, H, W] map owns neurons n with n // HW == c.  Give one
    # channel beta=0 (no memory) and check exactly its lanes lose their memory.
    B, C, HW, T = 2, 3, 4, 6
    N = C * HW
    rng = np.random.default_rng(8)
    I = rng.uniform(0.0, 0.4, (T, B * N))
    beta_c = np.array([0.9, 0.0, 0.9])
    lane_beta = O.lane_param(beta_c, B, N, "per_channel", C, HW)
    _, mem = O.leaky_forward(I, lane_beta, np.full(B * N, 1e30))
    ch = (np.arange(B * N) % N) // HW
    np.testing.assert_allclose(mem[:, ch == 1], I[:, ch == 1], atol=0)
    assert np.all(mem[1:, ch != 1] > I[1:, ch != 1])


def test_parameter_reductions_match_fd_on_shared_parameters():
    # A shared (scalar / per-channel / per-neuron) parameter's gradient is the
    # derivative with respect to that one shared value.
    B, C, HW, T = 2, 2, 3, 5
    N = C * HW
    rng = np.random.default_rng(9)
    I = rng.normal(0.6, 0.6, (T, B * N))
    gs = rng.normal(0, 1, (T, B * N))
    sg, k = "atan", 2.0
    for mode, size in (("scalar", 1), ("per_channel", C), ("per_neuron", N)):
        bp = rng.uniform(0.6, 0.9, size)
        tp = np.full(1, 1.0)

        def loss(bp_):
            lb = O.lane_param(bp_, B, N, mode, C, HW)
            lt = O.lane_param(tp, B, N, "scalar")
            spk, mem = O.leaky_forward(I, lb, lt, "none",
                                       spike_fn=lambda u: O.smooth_spike(u - lt, sg, k))
            return (gs * spk).sum(), spk, mem

        _, spk, mem = loss(bp)
        g = O.leaky_backward(mem, spk, gs, O.lane_param(bp, B, N, mode, C, HW),
                             O.lane_param(tp, B, N, "scalar"), "none", True, sg, k)
        red = O.reduce_lane_grad(g["grad_beta_lane"], B, N, mode, C, HW)
        h = 1e-6
        for j in range(size):
            bpp, bpm = bp.copy(), bp.copy()
            bpp[j] += h
            bpm[j] -= h
            np.testing.assert_allclose(red[j], (loss(bpp)[0] - loss(bpm)[0]) / (2 * h),
                                       rtol=1e-6, atol=1e-9)


# ---------------------------------------------------------------------------
# Library-backed pins: bfloat16 rounding, dense layer, cross-entropy
# ---------------------------------------------------------------------------

def test_bf16_round_matches_torch():
    rng = np.random.default_rng(10)
    x = np.concatenate([rng.normal(0, 3, 100000).astype(np.float32),
                        # exact ties between two bfloat16 neighbours
                        np.array([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -(1.0 + 2 ** -8),
                                  0.0, -0.0, 1e-40, 3.0e38], dtype=np.float32)])
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.bf16_round(x), ref)


def test_dense_forward_backward_match_torch():
    rng = np.random.default_rng(11)
    M, K, Nout = 37, 29, 13
    X = O.bf16_round(rng.normal(0, 1, (M, K)))
    W = O.bf16_round(rng.normal(0, 1, (Nout, K)))
    dI = rng.normal(0, 1, (M, Nout))
    tX, tW = torch.tensor(X, requires_grad=True), torch.tensor(W, requires_grad=True)
    out = tX @ tW.T
    out.backward(torch.tensor(dI))
    np.testing.assert_allclose(O.dense_forward(X, W), out.detach().numpy(), rtol=1e-13)
    dX, dW = O.dense_backward(X, W, dI)
    np.testing.assert_allclose(dX, tX.grad.numpy(), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dW, tW.grad.numpy(), rtol=1e-12, atol=1e-12)


def test_rate_ce_loss_matches_torch_autograd():
    rng = np.random.default_rng(12)
    T, B, C = 6, 9, 10
    spk = (rng.uniform(0, 1, (T, B, C)) < 0.3).astype(np.float64)
    y = rng.integers(0, C, B)
    loss, g = O.rate_ce_loss(spk, y)
    ts = torch.tensor(spk, requires_grad=True)
    ref = torch.nn.functional.cross_entropy(ts.sum(0), torch.tensor(y))
    ref.backward()
    assert abs(loss - ref.item()) < 1e-12
    np.testing.assert_allclose(g, ts.grad.numpy(), rtol=1e-12, atol=1e-14)


class _SpikeFastSigmoid(torch.autograd.Function):
    """Heaviside forward (Eq. 3) with the fast-sigmoid derivative of slope k
    in the backward: written directly in torch so that autograd, not the
    oracle's hand-written reverse recurrence, does the chain rule."""

    @staticmethod
    def forward(ctx, x, k):
        ctx.save_for_backward(x)
        ctx.k = k
        return (x > 0).to(x.dtype)

    @staticmethod
    def backward(ctx, g):
        (x,) = ctx.saved_tensors
        return g / (1.0 + ctx.k * x.abs()) ** 2, None


@pytest.mark.parametrize("k", [1.0, 5.0])
def test_dsnn_matches_torch_autograd(k):
    """The 3-layer dense SNN (dense -> Eq. 4 per layer, rate-coded CE) against
    a torch float64 network differentiated by autograd with the reset
    detached: spikes, loss and every dW agree."""
    rng = np.random.default_rng(13)
    T, B, sizes, beta, thr = 5, 4, (12, 9, 7, 5), 0.85, 1.0
    X = (rng.uniform(0, 1, (T * B, sizes[0])) < 0.4).astype(np.float64)
    Ws = [rng.uniform(-1.2, 1.2, (o, i)) for i, o in zip(sizes[:-1], sizes[1:])]
    y = rng.integers(0, sizes[-1], B)
    fwd = O.dsnn_forward(X, Ws, T, B, beta, thr, dtype=np.float64)
    res = O.dsnn_backward(fwd, Ws, y, T, B, beta, thr, k)

    tW = [torch.tensor(w, requires_grad=True) for w in Ws]
    x = torch.tensor(X)
    spikes = []
    for w in tW:
        cur = (x @ w.T).reshape(T, B, -1)
        u = torch.zeros(B, w.shape[0], dtype=torch.float64)
        z = torch.zeros_like(u)
        zs = []
        for t in range(T):
            u = beta * u + cur[t] - z.detach() * thr
            z = _SpikeFastSigmoid.apply(u - thr, k)
            zs.append(z)
        s = torch.stack(zs)
        spikes.append(s)
        x = s.reshape(T * B, -1)
    loss = torch.nn.functional.cross_entropy(spikes[-1].sum(0), torch.tensor(y))
    loss.backward()

    for l, s in enumerate(spikes):
        assert np.array_equal(fwd["spk"][l], s.detach().numpy().reshape(T, -1))
    assert all(0 < f.mean() < 1 for f in fwd["spk"])   # every layer spikes, not saturated
    assert abs(res["loss"] - loss.item()) < 1e-12
    for l, w in enumerate(tW):
        assert np.abs(w.grad.numpy()).max() > 1e-4      # a gradient reaches every layer
        np.testing.assert_allclose(res["dW"][l], w.grad.numpy(), rtol=1e-10, atol=1e-14)


def test_adamw_matches_torch_optim():
    """Three AdamW steps of the oracle against torch.optim.AdamW (the library
    routine) on float64 parameters."""
    rng = np.random.default_rng(14)
    n = 257
    w0 = rng.normal(0, 1, n)
    grads = [rng.normal(0, 1, n) * s for s in (1.0, 1e-3, 10.0)]
    lr, b1, b2, eps, wd = 1e-2, 0.9, 0.999, 1e-8, 0.05
    p = torch.tensor(w0, requires_grad=True)
    opt = torch.optim.AdamW([p], lr=lr, betas=(b1, b2), eps=eps, weight_decay=wd)
    w, m, v = w0.copy(), np.zeros(n), np.zeros(n)
    for k, g in enumerate(grads, start=1):
        p.grad = torch.tensor(g)
        opt.step()
        w, m, v = O.adamw_step(w, g, m, v, lr, b1, b2, eps, wd, k)
        np.testing.assert_allclose(w, p.detach().numpy(), rtol=1e-12, atol=1e-14)
    st = opt.state[p]
    np.testing.assert_allclose(m, st["exp_avg"].numpy(), rtol=1e-12)
    np.testing.assert_allclose(v, st["exp_avg_sq"].numpy(), rtol=1e-12)


# ---------------------------------------------------------------------------
# Recurrent Leaky neuron (Eq. 7)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("dtype,tol", [(np.float64, 1e-12), (np.float32, 1e-6)])
def test_hand_trace_rleaky(dtype, tol):
    # beta 0.5, thr 1, v 0.25: a spike feeds back v - thr = -0.75 at t+1.
    #  t0: 1.5 -> fire;  t1: 0.75 + 0.2 - 0.75 = 0.2;  t2: 0.1 + 1.0 = 1.1 -> fire;
    #  t3: 0.55 + 0 - 0.75 = -0.2;  t4: -0.1 + 0.9 = 0.8
    I = np.array([1.5, 0.2, 1.0, 0.0, 0.9])[:, None]
    spk, mem = O.rleaky_forward(I, [0.25], [0.5], [1.0], dtype=dtype)
    np.testing.assert_allclose(mem[:, 0], [1.5, 0.2, 1.1, -0.2, 0.8], rtol=tol, atol=tol)
    assert spk[:, 0].tolist() == [1, 0, 1, 0, 0]


def test_rleaky_special_cases_reduce_to_leaky():
    """v = 0 is the Leaky neuron with reset by subtraction; v = thr with the
    reset not detached is the Leaky neuron without reset (forward and
    BPTT); the recurrent weight's gradient is the reset term's with the
    opposite sign."""
    rng = np.random.default_rng(21)
    T, L = 9, 6
    I = rng.normal(0.6, 0.7, (T, L))
    beta, thr = rng.uniform(0.5, 0.95, L), rng.uniform(0.7, 1.2, L)
    gs, gm = rng.normal(0, 1, (T, L)), rng.normal(0, 0.5, (T, L))
    kw = dict(sg="atan", sg_param=2.0, grad_mem=gm)
    s0, m0 = O.rleaky_forward(I, np.zeros(L), beta, thr)
    s1, m1 = O.leaky_forward(I, beta, thr, "subtract")
    assert np.array_equal(s0, s1) and np.array_equal(m0, m1)
    for detach in (True, False):
        g0 = O.rleaky_backward(m0, s0, gs, np.zeros(L), beta, thr, detach=detach, **kw)
        g1 = O.leaky_backward(m1, s1, gs, beta, thr, "subtract", detach=detach, **kw)
        for k in ("grad_I", "grad_beta_lane", "grad_thr_lane", "grad_mem0"):
            np.testing.assert_allclose(g0[k], g1[k], rtol=1e-13, atol=1e-15)
    # following the free run's own spike path reproduces it
    zp = np.vstack([np.zeros((1, L)), s0[:-1]])
    s4, m4 = O.rleaky_forward(I, np.zeros(L), beta, thr, z_path=zp)
    assert np.array_equal(s4, s0) and np.array_equal(m4, m0)
    s2, m2 = O.rleaky_forward(I, thr, beta, thr)
    s3, m3 = O.leaky_forward(I, beta, thr, "none")
    assert np.array_equal(s2, s3)
    np.testing.assert_allclose(m2, m3, rtol=0, atol=1e-14)
    g2 = O.rleaky_backward(m2, s2, gs, thr, beta, thr, detach=False, **kw)
    g3 = O.leaky_backward(m3, s3, gs, beta, thr, "none", detach=False, **kw)
    np.testing.assert_allclose(g2["grad_I"], g3["grad_I"], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(g2["grad_beta_lane"], g3["grad_beta_lane"], rtol=1e-12, atol=1e-14)
    # thr enters both the spike and (v - thr): the none-reset thr gradient
    # plus the reset term's, which is -dv
    np.testing.assert_allclose(g2["grad_thr_lane"], g3["grad_thr_lane"] - g2["grad_v_lane"],
                               rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("detach", [True, False])
@pytest.mark.parametrize("sg,k", [("fast_sigmoid", 2.0), ("atan", 2.0)])
def test_rleaky_bptt_matches_finite_differences(detach, sg, k):
    rng = np.random.default_rng(31 + int(detach) + 2 * (sg == "atan"))
    T, L = 5, 3
    p = {"I": rng.normal(0.6, 0.6, (T, L)), "beta": rng.uniform(0.5, 0.95, L),
         "thr": rng.uniform(0.7, 1.2, L), "mem0": rng.normal(0.5, 0.5, L),
         "v": rng.uniform(-0.6, 0.6, L)}
    gs, gm, gmf = rng.normal(0, 1, (T, L)), rng.normal(0, 0.5, (T, L)), rng.normal(0, 1, L)
    f = lambda thr: (lambda u: O.smooth_spike(u - thr, sg, k))

    def loss(q, z_reset):
        spk, mem = O.rleaky_forward(q["I"], q["v"], q["beta"], q["thr"], mem0=q["mem0"],
                                    spike_fn=f(q["thr"]), z_reset=z_reset)
        return (gs * spk).sum() + (gm * mem).sum() + (gmf * mem[-1]).sum(), spk, mem

    _, spk, mem = loss(p, None)
    z_init = O.smooth_spike(p["mem0"] - p["thr"], sg, k)
    z_reset = np.vstack([z_init[None], spk[:-1]]) if detach else None
    g = O.rleaky_backward(mem, spk, gs, p["v"], p["beta"], p["thr"], detach=detach, sg=sg,
                          sg_param=k, grad_mem=gm, grad_mem_final=gmf, mem0=p["mem0"],
                          z_init=z_init)
    h = 1e-6

    def fd(name, idx):
        q = {kk: vv.copy() for kk, vv in p.items()}
        q[name][idx] += h
        lp = loss(q, z_reset)[0]
        q[name][idx] -= 2 * h
        return (lp - loss(q, z_reset)[0]) / (2 * h)

    for t in range(T):
        for l in range(L):
            np.testing.assert_allclose(g["grad_I"][t, l], fd("I", (t, l)), rtol=1e-6, atol=1e-8)
    for pname, gname in [("beta", "grad_beta_lane"), ("thr", "grad_thr_lane"),
                         ("mem0", "grad_mem0"), ("v", "grad_v_lane")]:
        for l in range(L):
            np.testing.assert_allclose(g[gname][l], fd(pname, l), rtol=1e-6, atol=1e-8)


def test_population_ce_matches_torch_autograd():
    """Population code (pop neurons per class, class-contiguous): the loss
    and spike gradient against torch's cross-entropy on population sums;
    pop = 1 is the plain readout."""
    rng = np.random.default_rng(15)
    T, B, C, pop = 1, 7, 10, 5
    spk = (rng.uniform(0, 1, (T, B, C * pop)) < 0.3).astype(np.float64)
    y = rng.integers(0, C, B)
    loss, g = O.rate_ce_loss(spk, y, pop)
    ts = torch.tensor(spk, requires_grad=True)
    counts = ts.sum(0).reshape(B, C, pop).sum(-1)
    ref = torch.nn.functional.cross_entropy(counts, torch.tensor(y))
    ref.backward()
    assert abs(loss - ref.item()) < 1e-12
    np.testing.assert_allclose(g, ts.grad.numpy(), rtol=1e-12, atol=1e-14)
    l1, g1 = O.rate_ce_loss(spk[:, :, :C], y, 1)
    l2, g2 = O.rate_ce_loss(spk[:, :, :C], y)
    assert l1 == l2 and np.array_equal(g1, g2)


# ---------------------------------------------------------------------------
# Convolutional SNN pieces (channel-last) against torch's NCHW operators
# ---------------------------------------------------------------------------

def test_conv2d_nhwc_matches_torch():
    rng = np.random.default_rng(16)
    X = rng.normal(0, 1, (3, 9, 11, 4))
    Wc = rng.normal(0, 1, (5, 3, 2, 4))
    tX = torch.tensor(X.transpose(0, 3, 1, 2), requires_grad=True)
    tW = torch.tensor(Wc.transpose(0, 3, 1, 2), requires_grad=True)
    y = torch.nn.functional.conv2d(tX, tW)
    dY = rng.normal(0, 1, y.shape)
    y.backward(torch.tensor(dY))
    np.testing.assert_allclose(O.conv2d_nhwc(X, Wc), y.detach().numpy().transpose(0, 2, 3, 1),
                               rtol=1e-12, atol=1e-12)
    dX, dW = O.conv2d_nhwc_backward(X, Wc, dY.transpose(0, 2, 3, 1))
    np.testing.assert_allclose(dX, tX.grad.numpy().transpose(0, 2, 3, 1), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dW, tW.grad.numpy().transpose(0, 2, 3, 1), rtol=1e-12, atol=1e-12)


def test_maxpool2_nhwc_matches_torch_including_ties():
    rng = np.random.default_rng(17)
    X = (rng.uniform(0, 1, (4, 6, 8, 3)) < 0.3).astype(np.float64)   # binary: many ties
    tX = torch.tensor(X.transpose(0, 3, 1, 2), requires_grad=True)
    y = torch.nn.functional.max_pool2d(tX, 2)
    dY = rng.normal(0, 1, y.shape)
    y.backward(torch.tensor(dY))
    Y, idx = O.maxpool2_nhwc(X)
    np.testing.assert_array_equal(Y, y.detach().numpy().transpose(0, 2, 3, 1))
    dX = O.maxpool2_nhwc_backward(dY.transpose(0, 2, 3, 1), idx, X.shape)
    np.testing.assert_array_equal(dX, tX.grad.numpy().transpose(0, 2, 3, 1))


def test_csnn_matches_torch_autograd():
    """The CSNN (conv -> Leaky with per-channel beta and reset to zero ->
    max pool, twice, then dense -> Leaky, rate-coded CE) against a torch
    float64 NCHW network differentiated by autograd with the reset
    detached: spikes, loss, every filter, the dense weights and the
    per-channel beta gradients agree."""
    rng = np.random.default_rng(18)
    T, B, k = 3, 2, 5.0
    X = (rng.uniform(0, 1, (T * B, 16, 16, 1)) < 0.4).astype(np.float64)
    convs = [rng.uniform(-1, 1, (3, 5, 5, 1)) * 0.6, rng.uniform(-1, 1, (4, 5, 5, 3)) * 0.5]
    # 16x16 -conv5-> 12x12 -pool-> 6x6 -conv5-> 2x2 -pool-> 1x1: 4 features
    Wfc = rng.uniform(-1, 1, (5, 4)) * 1.5
    betas = [rng.uniform(0.7, 0.95, 3), rng.uniform(0.7, 0.95, 4)]
    beta_fc, thr = 0.9, 1.0
    y = rng.integers(0, 5, B)
    fwd = O.csnn_forward(X, convs, Wfc, T, B, betas, beta_fc, thr, dtype=np.float64)
    res = O.csnn_backward(fwd, convs, Wfc, y, T, B, betas, beta_fc, thr, k)

    tconv = [torch.tensor(c.transpose(0, 3, 1, 2), requires_grad=True) for c in convs]
    tbeta = [torch.tensor(b, requires_grad=True) for b in betas]
    tfc = torch.tensor(Wfc, requires_grad=True)
    x = torch.tensor(X.transpose(0, 3, 1, 2))            # [T*B, C, H, W]
    spikes = []
    for wc, bc in zip(tconv, tbeta):
        cur = torch.nn.functional.conv2d(x, wc)
        C_, H_, W_ = cur.shape[1:]
        cur = cur.reshape(T, B, C_, H_, W_)
        u = torch.zeros(B, C_, H_, W_, dtype=torch.float64)
        z = torch.zeros_like(u)
        zs = []
        for t in range(T):
            u = bc.view(1, -1, 1, 1) * ((1 - z.detach()) * u) + cur[t]
            z = _SpikeFastSigmoid.apply(u - thr, k)
            zs.append(z)
        s = torch.stack(zs).reshape(T * B, C_, H_, W_)
        spikes.append(s)
        x = torch.nn.functional.max_pool2d(s, 2)
    flat = x.permute(0, 2, 3, 1).reshape(T * B, -1)      # channel-last flattening
    cur = (flat @ tfc.T).reshape(T, B, -1)
    u = torch.zeros(B, Wfc.shape[0], dtype=torch.float64)
    z = torch.zeros_like(u)
    zs = []
    for t in range(T):
        u = beta_fc * ((1 - z.detach()) * u) + cur[t]
        z = _SpikeFastSigmoid.apply(u - thr, k)
        zs.append(z)
    out = torch.stack(zs)
    loss = torch.nn.functional.cross_entropy(out.sum(0), torch.tensor(y))
    loss.backward()

    for l, s in enumerate(spikes):
        assert np.array_equal(fwd["spk"][l].reshape(-1), s.detach().numpy().transpose(0, 2, 3, 1).reshape(-1))
    assert np.array_equal(fwd["fc_spk"], out.detach().numpy().reshape(T, -1))
    assert all(0 < s.mean() < 1 for s in fwd["spk"])
    assert abs(res["loss"] - loss.item()) < 1e-12
    np.testing.assert_allclose(res["dW_fc"], tfc.grad.numpy(), rtol=1e-10, atol=1e-14)
    for l in range(2):
        assert np.abs(tconv[l].grad.numpy()).max() > 1e-6
        np.testing.assert_allclose(res["dW"][l], tconv[l].grad.numpy().transpose(0, 2, 3, 1),
                                   rtol=1e-10, atol=1e-14)
        np.testing.assert_allclose(res["dbeta"][l], tbeta[l].grad.numpy(), rtol=1e-10, atol=1e-14)
