"""CPU oracle for the spiking-neuron temporal scan — TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
legs of ``bench.py`` may import this module.  The CUDA library never calls it
and it never calls the CUDA library: the two share no code.

What it computes (arXiv 2211.10725, Sec. III-A and III-B):

* Eq. (3)  spike  z_t = 1 if u_t > u_thr else 0   (strict comparison)
* Eq. (4)  Leaky LIF with reset by subtraction
           u_t = beta*u_{t-1} + w x_t - z_{t-1}*u_thr
           (the input current I_t = w x_t is given; (1-beta) is absorbed in it)
* Eqs. (5)-(6) current-based (Synaptic) LIF
           i_t = alpha*i_{t-1} + I_t,   u_t = beta*u_{t-1} + i_t - z_{t-1}*u_thr
* Eq. (7)  recurrent Leaky LIF (one-to-one recurrent weight v)
           u_t = beta*u_{t-1} + w x_t + z_{t-1}*(v - u_thr)
* Eqs. (8)-(9) fast-sigmoid surrogate, and an arctan surrogate, substituted
  for dz/du in the backward pass (Sec. III-B).
* BPTT over the unrolled graph (Sec. II-A, II-B; Fig. 2): the exact reverse
  accumulation of the adjoint through the recurrences above, with the
  surrogate standing in for the Heaviside derivative.

Readings where the paper is silent (each is listed in the design notes):
reset-to-zero u_t = beta*(1-z_{t-1})*u_{t-1} + I_t (it clears only u in the
Synaptic neuron); the fast-sigmoid slope k gives dz/du <- 1/(1+k|u-thr|)^2
(k=1 is Eq. 9); arctan gives (a/2)/(1+(pi*a*(u-thr)/2)^2); a detached reset
treats z_{t-1} in the reset term as a constant; initial state u_{-1}=i_{-1}=0,
z_{-1}=0, or z_{-1}=[mem0 > thr] when mem0 is given; grad_mem_final is the
gradient of the loss with respect to the returned final state u_{T-1}; in
Eq. (7) a detached reset detaches only the -z*u_thr part: the recurrent
connection z*v always carries gradient.

Arrays are lane-major per time step: ``I[t, l]`` with lane l = b*N + n.  The
arithmetic runs in float64 unless ``dtype=np.float32`` is asked for; in that
mode each step is evaluated left to right as Eq. (4)/(6) are written
(beta*u, then + input, then - reset), one correctly rounded float32 operation
at a time.  That float32 evaluation is how a spike decision is taken in the
kernel's precision.

Everything here is deliberately plain: loops over t, numpy vector ops over
independent lanes, ``np.matmul`` for the dense layer.
"""
from __future__ import annotations

import math
from typing import Optional

import numpy as np

RESETS = ("subtract", "zero", "none")
SURROGATES = ("fast_sigmoid", "atan")
PARAM_MODES = ("scalar", "per_neuron", "per_channel")


# ---------------------------------------------------------------------------
# Parameters: scalar, per neuron [N] or per channel [C] -> one value per lane
# ---------------------------------------------------------------------------

def lane_param(p, B: int, N: int, mode: str, C: int = 1, HW: int = 1,
               dtype=np.float64) -> np.ndarray:
    """Expand a parameter to one value per lane l = b*N + n.

    per_channel: channel of neuron n is (n // HW) % C (N = C*H*W maps).
    """
    p = np.asarray(p, dtype=dtype).reshape(-1)
    n = np.arange(N)
    if mode == "scalar":
        per_n = np.full(N, p[0], dtype=dtype)
    elif mode == "per_neuron":
        per_n = p[n]
    elif mode == "per_channel":
        per_n = p[(n // HW) % C]
    else:
        raise ValueError(mode)
    return np.tile(per_n, B)


def reduce_lane_grad(g_lane: np.ndarray, B: int, N: int, mode: str, C: int = 1,
                     HW: int = 1) -> np.ndarray:
    """Sum per-lane parameter gradients into the parameter's own shape."""
    g = np.asarray(g_lane, dtype=np.float64).reshape(B, N)
    if mode == "scalar":
        return np.array([g.sum()])
    if mode == "per_neuron":
        return g.sum(axis=0)
    if mode == "per_channel":
        ch = (np.arange(N) // HW) % C
        out = np.zeros(C)
        for c in range(C):
            out[c] = g[:, ch == c].sum()
        return out
    raise ValueError(mode)


# ---------------------------------------------------------------------------
# Surrogate gradients (Sec. III-B, Eqs. 8-9)
# ---------------------------------------------------------------------------

def surrogate_grad(x: np.ndarray, kind: str, k: float) -> np.ndarray:
    """dz/du substitute evaluated at x = u - thr."""
    x = np.asarray(x, dtype=np.float64)
    if kind == "fast_sigmoid":
        return 1.0 / (1.0 + k * np.abs(x)) ** 2
    if kind == "atan":
        return (k / 2.0) / (1.0 + (math.pi * k * x / 2.0) ** 2)
    raise ValueError(kind)


def smooth_spike(x: np.ndarray, kind: str, k: float) -> np.ndarray:
    """The smooth function whose derivative is ``surrogate_grad`` (test-only
    forward used to check BPTT against finite differences): Eq. (8) with
    slope k, or 1/2 + atan(pi*k*x/2)/pi."""
    x = np.asarray(x, dtype=np.float64)
    if kind == "fast_sigmoid":
        return x / (1.0 + k * np.abs(x))
    if kind == "atan":
        return 0.5 + np.arctan(math.pi * k * x / 2.0) / math.pi
    raise ValueError(kind)


def heaviside(u: np.ndarray, thr: np.ndarray) -> np.ndarray:
    """Eq. (3): 1 where u > thr, else 0 (u == thr gives 0)."""
    return (u > thr).astype(u.dtype)


# ---------------------------------------------------------------------------
# Forward scans
# ---------------------------------------------------------------------------

def _initial(L, dtype, mem0, thr, spike):
    if mem0 is None:
        return np.zeros(L, dtype=dtype), np.zeros(L, dtype=dtype)
    u = np.asarray(mem0, dtype=dtype).reshape(L).copy()
    return u, spike(u)


def leaky_forward(I, beta, thr, reset: str = "subtract", mem0=None,
                  dtype=np.float64, spike_fn=None, z_reset=None):
    """Leaky LIF over T steps (Eqs. 3-4; reset-to-zero is the reading above).

    I: [T, L]; beta, thr: [L].  Returns (spk [T, L], mem [T, L]).

    spike_fn(u) replaces Eq. (3) (test-only smooth forward).  z_reset, if
    given as [T, L], supplies the constant z_{t-1} used by the reset term at
    step t as z_reset[t] (row 0 is z_{-1}): a detached reset held fixed.
    """
    I = np.asarray(I, dtype=dtype)
    T, L = I.shape
    beta = np.asarray(beta, dtype=dtype).reshape(L)
    thr = np.asarray(thr, dtype=dtype).reshape(L)
    spike = spike_fn if spike_fn is not None else (lambda u: heaviside(u, thr))
    u_prev, z_prev = _initial(L, dtype, mem0, thr, spike)
    spk = np.zeros((T, L), dtype=dtype)
    mem = np.zeros((T, L), dtype=dtype)
    for t in range(T):
        zr = z_prev if z_reset is None else np.asarray(z_reset[t], dtype=dtype)
        if reset == "subtract":
            u = beta * u_prev + I[t] - zr * thr
        elif reset == "zero":
            u = beta * ((1 - zr) * u_prev) + I[t]
        elif reset == "none":
            u = beta * u_prev + I[t]
        else:
            raise ValueError(reset)
        z = spike(u)
        mem[t], spk[t] = u, z
        u_prev, z_prev = u, z
    return spk, mem


def rleaky_forward(I, v, beta, thr, mem0=None, dtype=np.float64, spike_fn=None,
                   z_reset=None, z_path=None):
    """Recurrent Leaky LIF over T steps (Eqs. 3, 7): the spike of step t-1
    returns through the one-to-one weight v and the reset subtracts thr.

    I: [T, L]; v, beta, thr: [L].  Returns (spk [T, L], mem [T, L]).  Each
    step is (beta*u + I_t) + z_{t-1}*(v - thr), evaluated in ``dtype``.
    With z_reset (test-only), the reset part uses the given constant
    z_{t-1} while the recurrent part uses the live spike: u = beta*u + I_t +
    z_{t-1}*v - zr*thr.  With z_path ([T, L], row t = z_{t-1}; test-only)
    both parts follow the given spike sequence.
    """
    I = np.asarray(I, dtype=dtype)
    T, L = I.shape
    v = np.asarray(v, dtype=dtype).reshape(L)
    beta = np.asarray(beta, dtype=dtype).reshape(L)
    thr = np.asarray(thr, dtype=dtype).reshape(L)
    spike = spike_fn if spike_fn is not None else (lambda u: heaviside(u, thr))
    u_prev, z_prev = _initial(L, dtype, mem0, thr, spike)
    vmt = v - thr
    spk = np.zeros((T, L), dtype=dtype)
    mem = np.zeros((T, L), dtype=dtype)
    for t in range(T):
        if z_path is not None:
            u = beta * u_prev + I[t] + np.asarray(z_path[t], dtype=dtype) * vmt
        elif z_reset is None:
            u = beta * u_prev + I[t] + z_prev * vmt
        else:
            zr = np.asarray(z_reset[t], dtype=dtype)
            u = beta * u_prev + I[t] + z_prev * v - zr * thr
        z = spike(u)
        mem[t], spk[t] = u, z
        u_prev, z_prev = u, z
    return spk, mem


def synaptic_forward(I, alpha, beta, thr, reset: str = "subtract", mem0=None,
                     syn0=None, dtype=np.float64, spike_fn=None, z_reset=None):
    """Current-based LIF over T steps (Eqs. 3, 5, 6).

    Returns (spk, mem, syn), each [T, L].  Reset-to-zero clears only u.
    """
    I = np.asarray(I, dtype=dtype)
    T, L = I.shape
    alpha = np.asarray(alpha, dtype=dtype).reshape(L)
    beta = np.asarray(beta, dtype=dtype).reshape(L)
    thr = np.asarray(thr, dtype=dtype).reshape(L)
    spike = spike_fn if spike_fn is not None else (lambda u: heaviside(u, thr))
    u_prev, z_prev = _initial(L, dtype, mem0, thr, spike)
    i_prev = np.zeros(L, dtype=dtype) if syn0 is None else \
        np.asarray(syn0, dtype=dtype).reshape(L).copy()
    spk = np.zeros((T, L), dtype=dtype)
    mem = np.zeros((T, L), dtype=dtype)
    syn = np.zeros((T, L), dtype=dtype)
    for t in range(T):
        zr = z_prev if z_reset is None else np.asarray(z_reset[t], dtype=dtype)
        i = alpha * i_prev + I[t]
        if reset == "subtract":
            u = beta * u_prev + i - zr * thr
        elif reset == "zero":
            u = beta * ((1 - zr) * u_prev) + i
        elif reset == "none":
            u = beta * u_prev + i
        else:
            raise ValueError(reset)
        z = spike(u)
        syn[t], mem[t], spk[t] = i, u, z
        u_prev, z_prev, i_prev = u, z, i
    return spk, mem, syn


# ---------------------------------------------------------------------------
# BPTT (reverse-time accumulation of the adjoint)
# ---------------------------------------------------------------------------

def _bptt(mem, spk, grad_spk, beta, thr, reset, detach, sg, sg_param,
          grad_mem=None, grad_mem_final=None, mem0=None,
          syn=None, alpha=None, syn0=None, grad_syn_final=None, z_init=None, vrec=None):
    """Shared reverse pass for the Leaky (syn is None) and Synaptic neurons.

    The pass differentiates along the given trajectory (mem u_t, spk z_t),
    with z_t's dependence on u_t replaced by the surrogate.  Notation:
    du = dL/du_t (total), dz = dL/dz_t (total), di = dL/di_t (total).

      dz_t  = gs_t + [not detach] * (du_{t+1} * d u_{t+1} / d z_t)
      du_t  = gm_t + [t = T-1] gm_final + du_{t+1} * d u_{t+1}/d u_t
              + sigma'(u_t - thr) * dz_t
      di_t  = [t = T-1] gi_final + alpha * di_{t+1} + du_t         (Synaptic)
      dI_t  = du_t (Leaky) or di_t (Synaptic)

    with d u_{t+1}/d u_t = beta (subtract, none) or beta*(1-z_t) (zero) and
    d u_{t+1}/d z_t = -thr (subtract), -beta*u_t (zero), 0 (none).  The
    recurrent neuron (vrec = v, Eq. 7, subtract) adds v to d u_{t+1}/d z_t
    outside the detach factor, and dv += z_{t-1} * du_t.
    Parameter gradients, per lane, summed over t:
      dbeta  += du_t * d u_t/d beta   = du_t * u_{t-1}  (or (1-z_{t-1})*u_{t-1})
      dthr   += -sigma'_t * dz_t  -  [subtract] z_{t-1} * du_t
      dalpha += di_t * i_{t-1}
    Step t = -1 (the initial state) contributes through mem0 / syn0; its
    spike z_{-1} is [mem0 > thr] unless z_init gives the value the forward used.
    """
    mem = np.asarray(mem, dtype=np.float64)
    spk = np.asarray(spk, dtype=np.float64)
    gs = np.asarray(grad_spk, dtype=np.float64)
    T, L = mem.shape
    beta = np.asarray(beta, dtype=np.float64).reshape(L)
    thr = np.asarray(thr, dtype=np.float64).reshape(L)
    synaptic = syn is not None
    if synaptic:
        syn = np.asarray(syn, dtype=np.float64)
        alpha = np.asarray(alpha, dtype=np.float64).reshape(L)
    gm = None if grad_mem is None else np.asarray(grad_mem, dtype=np.float64)

    if mem0 is None:
        u_m1, z_m1, have_mem0 = np.zeros(L), np.zeros(L), False
    else:
        u_m1 = np.asarray(mem0, dtype=np.float64).reshape(L)
        z_m1 = (u_m1 > thr).astype(np.float64) if z_init is None else \
            np.asarray(z_init, dtype=np.float64).reshape(L)
        have_mem0 = True
    i_m1 = np.zeros(L) if (not synaptic or syn0 is None) else \
        np.asarray(syn0, dtype=np.float64).reshape(L)

    def u_at(t):
        return u_m1 if t < 0 else mem[t]

    def z_at(t):
        return z_m1 if t < 0 else spk[t]

    def decay(t):        # d u_{t+1} / d u_t
        return beta * (1.0 - z_at(t)) if reset == "zero" else beta

    def reset_slope(t):  # d u_{t+1} / d z_t
        if reset == "subtract":
            return -thr
        if reset == "zero":
            return -beta * u_at(t)
        return np.zeros(L)

    if vrec is not None:
        vrec = np.asarray(vrec, dtype=np.float64).reshape(L)
        dv = np.zeros(L)

    def rec_slope():     # d u_{t+1} / d z_t through the recurrent weight
        return vrec if vrec is not None else 0.0

    dI = np.zeros((T, L))
    dbeta = np.zeros(L)
    dthr = np.zeros(L)
    dalpha = np.zeros(L)
    du_next = np.zeros(L)
    di_next = np.zeros(L)
    for t in range(T - 1, -1, -1):
        s = surrogate_grad(mem[t] - thr, sg, sg_param)
        dz = gs[t] + ((0.0 if detach else 1.0) * reset_slope(t) + rec_slope()) * du_next
        du = decay(t) * du_next + s * dz
        if gm is not None:
            du = du + gm[t]
        if t == T - 1 and grad_mem_final is not None:
            du = du + np.asarray(grad_mem_final, dtype=np.float64).reshape(L)
        dthr += -s * dz
        if reset == "subtract":
            dthr += -z_at(t - 1) * du
        if vrec is not None:
            dv += z_at(t - 1) * du
        if reset == "zero":
            dbeta += du * (1.0 - z_at(t - 1)) * u_at(t - 1)
        else:
            dbeta += du * u_at(t - 1)
        if synaptic:
            di = alpha * di_next + du
            if t == T - 1 and grad_syn_final is not None:
                di = di + np.asarray(grad_syn_final, dtype=np.float64).reshape(L)
            dalpha += di * (syn[t - 1] if t > 0 else i_m1)
            dI[t] = di
            di_next = di
        else:
            dI[t] = du
        du_next = du

    # the initial state, step t = -1: z_{-1} depends on mem0 only if given
    dmem0 = decay(-1) * du_next
    if have_mem0:
        s = surrogate_grad(u_m1 - thr, sg, sg_param)
        dz = ((0.0 if detach else 1.0) * reset_slope(-1) + rec_slope()) * du_next
        dmem0 = dmem0 + s * dz
        dthr += -s * dz
    out = {"grad_I": dI, "grad_beta_lane": dbeta, "grad_thr_lane": dthr,
           "grad_mem0": dmem0}
    if synaptic:
        out["grad_alpha_lane"] = dalpha
        out["grad_syn0"] = alpha * di_next
    if vrec is not None:
        out["grad_v_lane"] = dv
    return out


def leaky_backward(mem, spk, grad_spk, beta, thr, reset="subtract", detach=True,
                   sg="fast_sigmoid", sg_param=25.0, grad_mem=None,
                   grad_mem_final=None, mem0=None, z_init=None):
    """BPTT for the Leaky neuron (Eq. 4) along the trajectory (mem, spk).

    Returns dict with grad_I [T,L], grad_beta_lane [L], grad_thr_lane [L],
    grad_mem0 [L] (all float64)."""
    return _bptt(mem, spk, grad_spk, beta, thr, reset, detach, sg, sg_param,
                 grad_mem, grad_mem_final, mem0, z_init=z_init)


def rleaky_backward(mem, spk, grad_spk, v, beta, thr, detach=True, sg="fast_sigmoid",
                    sg_param=25.0, grad_mem=None, grad_mem_final=None, mem0=None,
                    z_init=None):
    """BPTT for the recurrent Leaky neuron (Eq. 7) along (mem, spk).

    Adds grad_v_lane [L] to the Leaky outputs."""
    return _bptt(mem, spk, grad_spk, beta, thr, "subtract", detach, sg, sg_param,
                 grad_mem, grad_mem_final, mem0, z_init=z_init, vrec=v)


def synaptic_backward(mem, spk, syn, grad_spk, alpha, beta, thr, reset="subtract",
                      detach=True, sg="atan", sg_param=2.0, grad_mem=None,
                      grad_mem_final=None, mem0=None, syn0=None, grad_syn_final=None,
                      z_init=None):
    """BPTT for the current-based neuron (Eqs. 5-6) along (mem, spk, syn).

    Adds grad_alpha_lane [L] and grad_syn0 [L] to the Leaky outputs."""
    return _bptt(mem, spk, grad_spk, beta, thr, reset, detach, sg, sg_param,
                 grad_mem, grad_mem_final, mem0, syn=syn, alpha=alpha, syn0=syn0,
                 grad_syn_final=grad_syn_final, z_init=z_init)


# ---------------------------------------------------------------------------
# Dense layer (the synaptic operation w.x, Fig. 3) and rate-coded loss (Sec. V-A)
# ---------------------------------------------------------------------------

def bf16_round(x) -> np.ndarray:
    """Round float values to the nearest bfloat16 (ties to even), returned as
    float64.  Written from the bfloat16 format: keep the top 16 bits of the
    float32 pattern after adding half an ulp plus the tie-breaking bit."""
    f = np.asarray(x, dtype=np.float32)
    b = f.view(np.uint32).astype(np.uint64)
    lsb = (b >> 16) & 1
    r = ((b + 0x7FFF + lsb) >> 16) << 16
    out = r.astype(np.uint32).view(np.float32)
    nan = np.isnan(f)
    if nan.any():
        out = np.where(nan, np.float32("nan"), out)
    return out.astype(np.float64)


def dense_forward(X, W):
    """Input current I = X W^T over all T*B rows (float64 accumulation of the
    given operand values).  X: [M, K], W: [Nout, K]."""
    return np.matmul(np.asarray(X, np.float64), np.asarray(W, np.float64).T)


def dense_backward(X, W, dI):
    """dX = dI W and dW = dI^T X for I = X W^T."""
    X = np.asarray(X, np.float64)
    W = np.asarray(W, np.float64)
    dI = np.asarray(dI, np.float64)
    return np.matmul(dI, W), np.matmul(dI.T, X)


def rate_ce_loss(spk_out, labels, pop: int = 1):
    """Cross-entropy on output spike counts (rate-coded readout, Sec. V-A).

    spk_out: [T, B, C*pop] spikes; labels: [B].  With a population code
    (Sec. VII: pop output neurons per class, class c owning neurons
    c*pop .. c*pop + pop - 1), a class's count is the spikes of its whole
    population over all t.  Loss = mean_b CE(counts_b, y_b).
    Returns (loss, grad_spk [T, B, C*pop]) with grad = (softmax - onehot)/B
    of the neuron's class, at every t.
    """
    s = np.asarray(spk_out, dtype=np.float64)
    T, B, CP = s.shape
    C = CP // pop
    counts = s.sum(axis=0).reshape(B, C, pop).sum(axis=2)
    m = counts.max(axis=1, keepdims=True)
    lse = m[:, 0] + np.log(np.exp(counts - m).sum(axis=1))
    y = np.asarray(labels).astype(np.int64)
    loss = float(np.mean(lse - counts[np.arange(B), y]))
    p = np.exp(counts - lse[:, None])
    onehot = np.zeros((B, C))
    onehot[np.arange(B), y] = 1.0
    g = np.repeat((p - onehot) / B, pop, axis=1)
    return loss, np.broadcast_to(g, (T, B, CP)).copy()


# ---------------------------------------------------------------------------
# The dense SNN of Tab. I: dense layers feeding Leaky layers (Sec. V-A)
# ---------------------------------------------------------------------------

def dsnn_forward(X, Ws, T: int, B: int, beta: float, thr: float, dtype=np.float32):
    """Forward pass of a stack of dense -> Leaky layers.

    X: [T*B, K_0] input spikes (row t*B + b); Ws[l]: [N_l, K_l] with
    K_{l+1} = N_l.  Layer l: I_l = in_l W_l^T over all T*B rows
    (``dense_forward``, the synaptic operation of Fig. 3), then Eq. (4) with
    reset by subtraction over t (``leaky_forward``) in ``dtype``, the
    precision in which the spike decisions are taken; the spikes of layer l
    are the input of layer l + 1.

    Returns dict of per-layer lists: ``ins`` [T*B, K_l], ``I`` [T*B, N_l]
    (float64), ``spk`` and ``mem`` [T, B*N_l] (float64 copies of the
    ``dtype`` trace).
    """
    x = np.asarray(X, dtype=np.float64)
    out = {"ins": [], "I": [], "spk": [], "mem": []}
    for Wl in Ws:
        n = Wl.shape[0]
        I = dense_forward(x, Wl)
        L = B * n
        spk, mem = leaky_forward(I.astype(dtype).reshape(T, L), np.full(L, beta, dtype),
                                 np.full(L, thr, dtype), "subtract", dtype=dtype)
        out["ins"].append(x)
        out["I"].append(I)
        out["spk"].append(spk.astype(np.float64))
        out["mem"].append(mem.astype(np.float64))
        x = out["spk"][-1].reshape(T * B, n)
    return out


def dsnn_backward(fwd, Ws, labels, T: int, B: int, beta: float, thr: float,
                  sg_param: float, store=None, pop: int = 1):
    """Loss and BPTT of ``dsnn_forward``.

    The loss is ``rate_ce_loss`` on the last layer's spikes (``pop`` output
    neurons per class).  Then, from the
    top layer down: ``leaky_backward`` (detached reset, fast-sigmoid
    surrogate of slope ``sg_param``) on the layer's saved trace turns the
    spike gradient into dL/dI_l; ``dense_backward`` turns that into dL/dW_l
    and dL/din_l, which is the spike gradient of layer l - 1.

    ``store(x)`` rounds a value at each point where the path keeps it in a
    storage format (the loss gradient, every dL/dI_l and dL/din_l); None
    keeps float64 throughout.

    Returns dict: ``loss``, ``grad_out`` [T, B, C], and per-layer lists
    ``grad_spk`` [T, B*N_l], ``grad_I`` [T*B, N_l], ``dW`` [N_l, K_l].
    """
    keep = (lambda a: a) if store is None else store
    nl = len(Ws)
    C = Ws[-1].shape[0]   # output neurons (classes * pop)
    loss, g_out = rate_ce_loss(fwd["spk"][-1].reshape(T, B, C), labels, pop)
    g_out = keep(g_out)
    gs = g_out.reshape(T, B * C)
    res = {"loss": loss, "grad_out": g_out, "grad_spk": [None] * nl,
           "grad_I": [None] * nl, "dW": [None] * nl}
    for l in range(nl - 1, -1, -1):
        n = Ws[l].shape[0]
        L = B * n
        res["grad_spk"][l] = gs
        g = leaky_backward(fwd["mem"][l], fwd["spk"][l], gs, np.full(L, beta), np.full(L, thr),
                           reset="subtract", detach=True, sg="fast_sigmoid", sg_param=sg_param)
        dI = keep(g["grad_I"]).reshape(T * B, n)
        dX, dW = dense_backward(fwd["ins"][l], Ws[l], dI)
        res["grad_I"][l] = dI
        res["dW"][l] = dW
        gs = keep(dX).reshape(T, B * Ws[l].shape[1])
    return res


# ---------------------------------------------------------------------------
# Optimiser of the training runs (Sec. V): AdamW
# ---------------------------------------------------------------------------

def adamw_step(w, g, m, v, lr, beta1, beta2, eps, weight_decay, step):
    """One AdamW update (Adam with decoupled weight decay, Loshchilov and
    Hutter): moment estimates, their bias corrections 1 - beta^step, and a
    decay of w by lr * weight_decay applied beside the Adam step.  Float64.
    Returns (w, m, v)."""
    w, g, m, v = (np.asarray(a, dtype=np.float64) for a in (w, g, m, v))
    m = beta1 * m + (1.0 - beta1) * g
    v = beta2 * v + (1.0 - beta2) * g * g
    m_hat = m / (1.0 - beta1 ** step)
    v_hat = v / (1.0 - beta2 ** step)
    w = w - lr * weight_decay * w - lr * m_hat / (np.sqrt(v_hat) + eps)
    return w, m, v


# ---------------------------------------------------------------------------
# The convolutional SNN of Tab. I (CSNN): 5x5 convolutions and 2x2 max
# pooling around Leaky layers, channel-last activations [M, H, W, C]
# ---------------------------------------------------------------------------

def conv2d_nhwc(X, Wc):
    """Valid 2-D convolution (stride 1) of X [M, H, W, Cin] with filters
    Wc [Cout, KH, KW, Cin]: Y[m, y, x, o] = sum_{ky,kx,c} X[m, y+ky, x+kx, c]
    * Wc[o, ky, kx, c] (float64).  Returns [M, H-KH+1, W-KW+1, Cout]."""
    X = np.asarray(X, np.float64)
    Wc = np.asarray(Wc, np.float64)
    KH, KW = Wc.shape[1], Wc.shape[2]
    win = np.lib.stride_tricks.sliding_window_view(X, (KH, KW), axis=(1, 2))
    # win: [M, Ho, Wo, Cin, KH, KW]
    return np.einsum("mhwcij,oijc->mhwo", win, Wc)


def conv2d_nhwc_backward(X, Wc, dY):
    """Gradients of conv2d_nhwc: dX [M, H, W, Cin] (each output gradient
    spread back over the input window it read) and dW [Cout, KH, KW, Cin]."""
    X = np.asarray(X, np.float64)
    Wc = np.asarray(Wc, np.float64)
    dY = np.asarray(dY, np.float64)
    KH, KW = Wc.shape[1], Wc.shape[2]
    Ho, Wo = dY.shape[1], dY.shape[2]
    win = np.lib.stride_tricks.sliding_window_view(X, (KH, KW), axis=(1, 2))
    dW = np.einsum("mhwo,mhwcij->oijc", dY, win)
    dX = np.zeros_like(X)
    for ky in range(KH):
        for kx in range(KW):
            dX[:, ky:ky + Ho, kx:kx + Wo, :] += np.einsum("mhwo,oc->mhwc", dY, Wc[:, ky, kx, :])
    return dX, dW


def maxpool2_nhwc(X):
    """2x2 max pooling with stride 2 of X [M, H, W, C] (H, W even).  Returns
    (Y [M, H/2, W/2, C], idx) where idx is the window position (0..3, row
    major) of the first maximum, which the backward routes the gradient to."""
    X = np.asarray(X, np.float64)
    M, H, W, C = X.shape
    w = X.reshape(M, H // 2, 2, W // 2, 2, C).transpose(0, 1, 3, 5, 2, 4).reshape(
        M, H // 2, W // 2, C, 4)
    idx = np.argmax(w, axis=-1)   # first maximum in window order
    return np.take_along_axis(w, idx[..., None], -1)[..., 0], idx


def maxpool2_nhwc_backward(dY, idx, shape):
    """Gradient of maxpool2_nhwc: dY to the window position idx, 0 elsewhere."""
    M, H, W, C = shape
    d = np.zeros((M, H // 2, W // 2, C, 4))
    np.put_along_axis(d, np.asarray(idx)[..., None], np.asarray(dY, np.float64)[..., None], -1)
    return d.reshape(M, H // 2, W // 2, C, 2, 2).transpose(0, 1, 4, 2, 5, 3).reshape(M, H, W, C)


def csnn_forward(X, convs, Wfc, T: int, B: int, beta_convs, beta_fc: float, thr: float,
                 reset: str = "zero", dtype=np.float32):
    """Forward pass of the CSNN: per conv layer conv2d_nhwc, a Leaky layer
    (Eq. 4 with the given reset, per-channel beta) over t, maxpool2_nhwc;
    then a dense layer (the flattened [H, W, C] map) and a Leaky output
    layer.  X: [T*B, H, W, Cin] input spikes; convs: list of [Cout, KH, KW,
    Cin] filters; Wfc [Nout, H*W*C]; beta_convs: per-channel betas (one
    array per conv layer).  Spike decisions in ``dtype``.

    Returns a dict of per-layer lists: ``ins`` (layer input), ``I`` (input
    current, float64), ``spk``/``mem`` ([T, B*N], N = H*W*C), ``pool`` (the
    pooled spikes) and ``idx`` (pooling positions)."""
    x = np.asarray(X, np.float64)
    out = {"ins": [], "I": [], "spk": [], "mem": [], "pool": [], "idx": []}
    for Wc, bc in zip(convs, beta_convs):
        I = conv2d_nhwc(x, Wc)
        Mq, Ho, Wo, Co = I.shape
        L = B * Ho * Wo * Co
        beta = np.tile(np.asarray(bc, np.float64), B * Ho * Wo)  # channel-last lanes
        spk, mem = leaky_forward(I.astype(dtype).reshape(T, L), beta.astype(dtype),
                                 np.full(L, thr, dtype), reset, dtype=dtype)
        s = spk.astype(np.float64).reshape(T * B, Ho, Wo, Co)
        p, idx = maxpool2_nhwc(s)
        for k, v in (("ins", x), ("I", I), ("spk", spk.astype(np.float64)),
                     ("mem", mem.astype(np.float64)), ("pool", p), ("idx", idx)):
            out[k].append(v)
        x = p
    flat = x.reshape(T * B, -1)
    I = dense_forward(flat, Wfc)
    n = Wfc.shape[0]
    spk, mem = leaky_forward(I.astype(dtype).reshape(T, B * n), np.full(B * n, beta_fc, dtype),
                             np.full(B * n, thr, dtype), reset, dtype=dtype)
    out["fc_in"], out["fc_I"] = flat, I
    out["fc_spk"], out["fc_mem"] = spk.astype(np.float64), mem.astype(np.float64)
    return out


def csnn_backward(fwd, convs, Wfc, labels, T: int, B: int, beta_convs, beta_fc: float,
                  thr: float, sg_param: float, reset: str = "zero", store=None):
    """Loss and BPTT of ``csnn_forward``: rate_ce_loss on the output spikes;
    the output layer's BPTT and dense backward; then per conv layer from
    the top the max-pool backward, the Leaky BPTT (detached reset,
    fast-sigmoid slope ``sg_param``; per-channel beta gradients) and the
    convolution backward.  ``store`` rounds where the path keeps a value in
    a storage format (as in dsnn_backward).

    Returns dict: loss, dW_fc, dW (per conv layer), dbeta (per conv layer,
    per channel), and the gradients of every stage (grad_out, grad_I_fc,
    grad_pool, grad_I)."""
    keep = (lambda a: a) if store is None else store
    n = Wfc.shape[0]
    loss, g_out = rate_ce_loss(fwd["fc_spk"].reshape(T, B, n), labels)
    g_out = keep(g_out)
    g = leaky_backward(fwd["fc_mem"], fwd["fc_spk"], g_out.reshape(T, B * n),
                       np.full(B * n, beta_fc), np.full(B * n, thr), reset=reset, detach=True,
                       sg="fast_sigmoid", sg_param=sg_param)
    dI_fc = keep(g["grad_I"]).reshape(T * B, n)
    d_flat, dW_fc = dense_backward(fwd["fc_in"], Wfc, dI_fc)
    res = {"loss": loss, "grad_out": g_out, "grad_I_fc": dI_fc, "dW_fc": dW_fc,
           "dW": [None] * len(convs), "dbeta": [None] * len(convs),
           "grad_pool": [None] * len(convs), "grad_I": [None] * len(convs)}
    d_pool = keep(d_flat).reshape(fwd["pool"][-1].shape)
    for l in range(len(convs) - 1, -1, -1):
        res["grad_pool"][l] = d_pool
        s_shape = fwd["I"][l].shape
        Mq, Ho, Wo, Co = s_shape
        d_spk = maxpool2_nhwc_backward(d_pool, fwd["idx"][l], s_shape)
        L = B * Ho * Wo * Co
        beta = np.tile(np.asarray(beta_convs[l], np.float64), B * Ho * Wo)
        g = leaky_backward(fwd["mem"][l], fwd["spk"][l], d_spk.reshape(T, L), beta,
                           np.full(L, thr), reset=reset, detach=True, sg="fast_sigmoid",
                           sg_param=sg_param)
        dI = keep(g["grad_I"]).reshape(T * B, Ho, Wo, Co)
        res["grad_I"][l] = dI
        res["dbeta"][l] = reduce_lane_grad(g["grad_beta_lane"], B, Ho * Wo * Co, "per_channel",
                                           C=Co, HW=1)
        dX, dW = conv2d_nhwc_backward(fwd["ins"][l], convs[l], dI)
        res["dW"][l] = dW
        if l > 0:
            d_pool = keep(dX)
    return res
