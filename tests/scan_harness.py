"""Helpers shared by the scan parity tests: run the CPU oracle on the seeded
inputs of a workload and compare the CUDA results with it.

Comparison protocol
-------------------
* Spike decisions are integers decided by floating point, so both sides take
  them in the kernel's precision: the oracle's float32 evaluation of Eqs.
  (4)/(6) (``dtype=np.float32``) gives the expected spike train and membrane
  trace, and the GPU must reproduce both bit for bit.
* That float32 trace is pinned to the float64 definition: the oracle reruns
  the scan in float64 with the reset sequence held at the float32 spikes, and
  every element where the float64 spike would differ must lie within 1e-5 of
  the threshold (the only places where several answers are correct); mem
  agrees within rel 1e-5 / abs 1e-6.
* The backward is a function of the saved forward state (mem, spk): the
  oracle's float64 BPTT runs on the same saved state the kernel consumes
  (the float32 trace, rounded to the storage dtype in the store variant) and
  the kernel's gradients must agree within the stated tolerances.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import snn_oracle as O
from paper_2211_10725_gb300 import workloads as W

TOL = {  # (rtol, atol) for values compared elementwise
    W.F32: (1e-5, 1e-6),
    W.BF16: (2e-2, 1e-3),
    W.F16: (2e-2, 1e-3),
}
AMBIGUITY = 1e-5   # |u - thr| below which a spike decision may legitimately differ


def lanes_2d(x: torch.Tensor, lanes=None) -> np.ndarray:
    """[T, B, N] tensor (any dtype, any device) -> float64 [T, L'] array
    (the lanes are taken before the conversion)."""
    a = x.detach().to("cpu")
    a = a.reshape(a.shape[0], -1)
    if lanes is not None:
        a = a[:, torch.from_numpy(np.asarray(lanes, dtype=np.int64))]
    return a.to(torch.float32).numpy().astype(np.float64)


def lanes_1d(x, lanes=None) -> np.ndarray:
    a = x.detach().to("cpu").reshape(-1)
    if lanes is not None:
        a = a[torch.from_numpy(np.asarray(lanes, dtype=np.int64))]
    return a.to(torch.float32).numpy().astype(np.float64)


class HostCopy:
    """The outputs of a ScanLayer copied to host memory once, with the same
    attribute names, so that many lane blocks can be compared without a
    device transfer each."""

    NAMES = ("spk", "mem", "syn", "mem_final", "grad_I", "grad_mem0", "grad_syn0", "grad_beta",
             "grad_thr", "grad_alpha", "grad_v")

    def __init__(self, layer):
        for k in self.NAMES:
            v = getattr(layer, k, None)
            setattr(self, k, None if v is None else v.detach().cpu())


def round_to(dtype: str, x: np.ndarray) -> np.ndarray:
    """Round to the storage dtype (library conversion, round to nearest even)."""
    if dtype == W.F32:
        return np.asarray(x, dtype=np.float32).astype(np.float64)
    t = torch.from_numpy(np.asarray(x, dtype=np.float32)).to(W.TORCH_DTYPE[dtype])
    return t.to(torch.float32).numpy().astype(np.float64)


def oracle_expect(w: W.ScanWorkload, inp: dict, lanes=None, backward=True) -> dict:
    """Oracle results for the workload's inputs on a subset of lanes."""
    T, B, N, C, HW = w.T, w.B, w.N, w.C, w.HW
    L = B * N
    idx = np.arange(L) if lanes is None else np.asarray(lanes)
    syn = w.neuron == "synaptic"
    rec = w.neuron == "rleaky"

    def par(name, mode):
        full = O.lane_param(inp[name].numpy(), B, N, mode, C, HW)
        return full[idx]

    beta, thr = par("beta", w.beta_mode), par("thr", w.thr_mode)
    alpha = par("alpha", w.alpha_mode) if syn else None
    v = par("v", w.v_mode) if rec else None
    I = lanes_2d(inp["I"], idx)
    mem0 = lanes_1d(inp["mem0"], idx) if "mem0" in inp else None
    syn0 = lanes_1d(inp["syn0"], idx) if "syn0" in inp else None
    f32 = lambda a: None if a is None else np.asarray(a, dtype=np.float32)

    # float32 evaluation: the spike decisions in the kernel's precision
    if syn:
        spk32, mem32, syn32 = O.synaptic_forward(f32(I), f32(alpha), f32(beta), f32(thr), w.reset,
                                                 mem0=f32(mem0), syn0=f32(syn0), dtype=np.float32)
    elif rec:
        spk32, mem32 = O.rleaky_forward(f32(I), f32(v), f32(beta), f32(thr), mem0=f32(mem0),
                                        dtype=np.float32)
        syn32 = None
    else:
        spk32, mem32 = O.leaky_forward(f32(I), f32(beta), f32(thr), w.reset, mem0=f32(mem0),
                                       dtype=np.float32)
        syn32 = None
    z_m1 = np.zeros(len(idx)) if mem0 is None else (f32(mem0) > f32(thr)).astype(np.float64)
    z_reset = np.vstack([z_m1[None], spk32[:-1].astype(np.float64)]) if T > 0 else None

    # float64 scan on the same discrete path (reset held at the fp32 spikes)
    if syn:
        _, mem64, syn64 = O.synaptic_forward(I, alpha, beta, thr, w.reset, mem0=mem0, syn0=syn0,
                                             z_reset=z_reset)
    elif rec:
        _, mem64 = O.rleaky_forward(I, v, beta, thr, mem0=mem0, z_path=z_reset)
        syn64 = None
    else:
        _, mem64 = O.leaky_forward(I, beta, thr, w.reset, mem0=mem0, z_reset=z_reset)
        syn64 = None
    out = {"lanes": idx, "spk32": spk32.astype(np.float64), "mem32": mem32.astype(np.float64),
           "mem64": mem64, "thr": thr, "beta": beta, "alpha": alpha, "v": v, "I": I,
           "mem0": mem0, "syn0": syn0, "reset": w.reset}
    if syn:
        out["syn32"], out["syn64"] = syn32.astype(np.float64), syn64
    if not backward:
        return out

    # backward on the saved state as the kernel consumes it
    gs = lanes_2d(inp["grad_spk"], idx)
    gm = lanes_2d(inp["grad_mem"], idx) if "grad_mem" in inp else None
    gmf = lanes_1d(inp["grad_mem_final"], idx) if "grad_mem_final" in inp else None
    gsf = lanes_1d(inp["grad_syn_final"], idx) if "grad_syn_final" in inp else None
    mem_b = out["mem32"] if w.save == "recompute" else round_to(w.io_dtype, out["mem32"])
    kw = dict(reset=w.reset, detach=w.detach_reset, sg=w.surrogate, sg_param=w.sg_param,
              grad_mem=gm, grad_mem_final=gmf, mem0=mem0)
    if syn:
        syn_b = out["syn32"] if w.save == "recompute" else round_to(w.io_dtype, out["syn32"])
        g = O.synaptic_backward(mem_b, out["spk32"], syn_b, gs, alpha, beta, thr, syn0=syn0,
                                grad_syn_final=gsf, **kw)
    elif rec:
        kr = {k: kw[k] for k in kw if k != "reset"}
        g = O.rleaky_backward(mem_b, out["spk32"], gs, v, beta, thr, **kr)
    else:
        g = O.leaky_backward(mem_b, out["spk32"], gs, beta, thr, **kw)
    out.update(g)
    # magnitude of the terms each gradient sums: the same reverse recurrence
    # on absolute upstream gradients (all coefficients are then >= 0), so fp32
    # accumulation error can be judged against it where the result cancels
    ab = lambda a: None if a is None else np.abs(a)
    kwa = dict(kw, detach=True, grad_mem=ab(gm), grad_mem_final=ab(gmf))
    if syn:
        ga = O.synaptic_backward(mem_b, out["spk32"], syn_b, np.abs(gs), alpha, beta, thr,
                                 syn0=syn0, grad_syn_final=ab(gsf), **kwa)
        out["grad_syn0_scale"] = np.maximum(ga["grad_syn0"], np.abs(g["grad_syn0"]))
    elif rec:
        # |v| (+ thr for a live reset) as the spike's coefficient keeps every
        # term of the absolute-value pass non-negative
        va = np.abs(v) + (0.0 if w.detach_reset else np.abs(thr))
        kra = {k: kwa[k] for k in kwa if k != "reset"}
        ga = O.rleaky_backward(mem_b, out["spk32"], np.abs(gs), va, beta, thr, **kra)
    else:
        ga = O.leaky_backward(mem_b, out["spk32"], np.abs(gs), beta, thr, **kwa)
    out["grad_I_scale"] = np.maximum(ga["grad_I"], np.abs(g["grad_I"]))
    out["grad_mem0_scale"] = np.maximum(np.abs(ga["grad_mem0"]), np.abs(g["grad_mem0"]))
    if lanes is None:
        out["grad_beta"] = O.reduce_lane_grad(g["grad_beta_lane"], B, N, w.beta_mode, C, HW)
        out["grad_thr"] = O.reduce_lane_grad(g["grad_thr_lane"], B, N, w.thr_mode, C, HW)
        if syn:
            out["grad_alpha"] = O.reduce_lane_grad(g["grad_alpha_lane"], B, N, w.alpha_mode, C, HW)
        if rec:
            out["grad_v"] = O.reduce_lane_grad(g["grad_v_lane"], B, N, w.v_mode, C, HW)
    return out


EPS32 = 2.0 ** -24


def fp32_trace_bound(ref) -> tuple:
    """Running first-order bound on |u32 - u64| (and |i32 - i64|) for the
    float32 evaluation of Eqs. (4)-(6) along the same spike path: each step
    adds at most one rounding (relative EPS32) per operation to the carried
    error, which decays by beta (alpha) per step."""
    u64, T = ref["mem64"], ref["mem64"].shape[0]
    L = u64.shape[1]
    beta, alpha = ref["beta"], ref["alpha"]
    syn = "syn64" in ref
    z = ref["spk32"]
    eu, ei = np.zeros(L), np.zeros(L)
    bu, bi = np.zeros((T, L)), np.zeros((T, L))
    u_prev = np.zeros(L) if ref["mem0"] is None else ref["mem0"]
    z_prev = np.zeros(L) if ref["mem0"] is None else (ref["mem0"] > ref["thr"]).astype(float)
    i_prev = np.zeros(L) if ref.get("syn0") is None else ref["syn0"]
    for t in range(T):
        x = ref["I"][t]
        if syn:
            i = ref["syn64"][t]
            ei = alpha * ei + EPS32 * (np.abs(alpha * i_prev) + np.abs(i))
            bi[t] = ei
            x, i_prev = i, i
        keep = (1.0 - z_prev) if ref["reset"] == "zero" else 1.0
        decayed = beta * keep * u_prev
        eu = beta * keep * eu + (ei if syn else 0.0) + EPS32 * (
            np.abs(decayed) + np.abs(decayed + x) + np.abs(u64[t]))
        if ref.get("v") is not None:  # v - thr is rounded once in fp32
            eu = eu + z_prev * EPS32 * np.abs(ref["v"] - ref["thr"])
        bu[t] = eu
        u_prev, z_prev = u64[t], z[t]
    return bu, bi


def check_spikes_and_mem(w, ref, spk_gpu, mem_gpu=None, syn_gpu=None, lanes=None):
    """Bit-exact spikes and trace against the fp32 evaluation; fp32 trace
    within its rounding bound of the float64 scan on the same spike path."""
    spk = lanes_2d(spk_gpu, lanes)
    mism = np.argwhere(spk != ref["spk32"])
    assert mism.size == 0, f"{len(mism)} spike mismatches, first at {mism[:5].tolist()}"
    bu, bi = fp32_trace_bound(ref)
    # the fp32 spike path is a valid one: the float64 decision differs only
    # where u is within AMBIGUITY (or the fp32 rounding bound) of the threshold
    z64 = (ref["mem64"] > ref["thr"][None]).astype(np.float64)
    diff = z64 != ref["spk32"]
    if diff.any():
        margin = np.abs(ref["mem64"] - ref["thr"][None])[diff]
        allowed = np.maximum(AMBIGUITY, 2.0 * bu[diff])
        assert np.all(margin < allowed), f"fp32 spike off the fp64 path by {margin.max()}"
    n_mem = assert_close("mem32 vs mem64", ref["mem32"], ref["mem64"], 1e-5,
                         np.maximum(1e-6, 2.0 * bu))
    if mem_gpu is not None:
        m = lanes_2d(mem_gpu, lanes)
        expect = round_to(w.io_dtype, ref["mem32"])
        bad = np.argwhere(m != expect)
        assert bad.size == 0, f"{len(bad)} mem mismatches, first {bad[:5].tolist()}"
    if syn_gpu is not None:
        s = lanes_2d(syn_gpu, lanes)
        expect = round_to(w.io_dtype, ref["syn32"])
        assert np.array_equal(s, expect)
        n_mem += assert_close("syn32 vs syn64", ref["syn32"], ref["syn64"], 1e-5,
                              np.maximum(1e-6, 2.0 * bi))
    return {"spk_fp64_ambiguous": int(diff.sum()), "mem_fp32_bound": n_mem}


def assert_close(name, got, ref, rtol, atol, scale=None):
    """|got - ref| <= atol + rtol * scale, scale = |ref| unless given (the
    magnitude of the terms a computed sum accumulates).

    Returns the number of elements that pass only through the widened band:
    beyond atol + rtol * |ref| but within the limit (0 without `scale` or an
    array-valued atol wider than its scalar floor)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    err = np.abs(got - ref)
    lim = atol + rtol * (np.abs(ref) if scale is None else scale)
    bad = err > lim
    if bad.any():
        i = np.unravel_index(np.argmax(err - lim), err.shape)
        raise AssertionError(f"{name}: {bad.sum()} / {bad.size} beyond tolerance; worst at {i}: "
                             f"got {got[i]!r} ref {ref[i]!r} (rtol {rtol}, atol {atol})")
    plain = np.min(atol) + rtol * np.abs(ref)
    return int(np.count_nonzero(err > plain))


def assert_widened(counts: dict, sizes: dict, frac: float = 1e-3):
    """Print how many elements of each compared output were judged by a
    widened band (spikes off the float64 decision within the ambiguity
    band, trace values beyond rel 1e-5 but within the float32 rounding
    bound, gradients beyond rel tol of |ref| but within the tolerance of
    the summed terms' magnitude), and assert each is at most `frac` of the
    output's elements (plus 2, for outputs of a few elements); the initial
    state's gradients (a sum over every step, where a recurrent neuron's
    terms can grow large and cancel) at most 10 * `frac`."""
    for k, n in counts.items():
        total = max(1, sizes.get(k, 1))
        f = 10 * frac if k in ("grad_mem0", "grad_syn0") else frac
        print(f"widened {k}: {n} of {total}")
        assert n <= f * total + 2, f"{k}: {n} of {total} elements judged by a widened band"


def check_param_grad(name, got, ref, lane_partials, B, N, mode, C, HW, rtol=1e-5):
    """A reduced parameter gradient: relative to its value, with an absolute
    floor proportional to the sum of |per-lane partials| it reduces (fp32
    accumulation over t within a lane, fp64 across lanes).  Returns the
    count judged by that floor."""
    scale = O.reduce_lane_grad(np.abs(lane_partials), B, N, mode, C, HW)
    return assert_close(name, got, ref, rtol, rtol * scale + 1e-6)


def run_gpu(w: W.ScanWorkload, inp: dict, device="cuda", **desc_over):
    """Forward + backward of one workload through the C ABI; returns the
    ScanLayer holding every output (on the device)."""
    from paper_2211_10725_gb300 import snn
    d = {k: v.to(device) for k, v in inp.items()}
    layer = snn.ScanLayer(w, device=device, want_syn=True, **desc_over)
    layer.forward(d["I"], d["beta"], d["thr"], d.get("alpha"), d.get("mem0"), d.get("syn0"),
                  v=d.get("v"))
    layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], alpha=d.get("alpha"),
                   mem0=d.get("mem0"), syn0=d.get("syn0"), grad_mem=d.get("grad_mem"),
                   grad_mem_final=d.get("grad_mem_final"),
                   grad_syn_final=d.get("grad_syn_final"), v=d.get("v"))
    torch.cuda.synchronize()
    return layer


FMAX = {W.F32: float(np.finfo(np.float32).max), W.BF16: 3.3895313892515355e38,
        W.F16: 65504.0}


def overflow_mask(g_ref, dtype):
    """Where the float64 reverse pass leaves the storage dtype's range: per
    lane, every step from the last one (the reverse pass runs from t = T-1
    down) at which |dL/dI| exceeds the largest finite value, and before it.
    Returns (mask [T, L'], lanes [L'])."""
    big = np.abs(g_ref) > FMAX[dtype]
    lanes = big.any(axis=0)
    if not lanes.any():
        return np.zeros_like(big), lanes
    T = g_ref.shape[0]
    t_over = np.where(lanes, T - 1 - np.argmax(big[::-1], axis=0), -1)
    return np.arange(T)[:, None] <= t_over[None, :], lanes


def extreme_lanes(g_ref):
    """Lanes whose float64 reverse pass comes within a factor 1e3 of the
    fp32 range: their per-lane fp32 sums over t (parameter partials, the
    initial state's gradient) can overflow part-way even where the exact
    result is finite, so they have no fp32 value to compare."""
    return (np.abs(g_ref) > 1e-3 * FMAX[W.F32]).any(axis=0)


def check_overflow(name, got, ref, mask, dtype):
    """At the step where a lane's gradient first leaves the range (in the
    reverse pass's order) the GPU must hold the same-signed infinity; the
    earlier steps of such a lane have no value in the storage dtype and are
    not compared."""
    T = ref.shape[0]
    big = np.abs(ref) > FMAX[dtype]
    lanes = big.any(axis=0)
    t_over = T - 1 - np.argmax(big[::-1], axis=0)
    idx = np.nonzero(lanes)[0]
    g = got[t_over[idx], idx]
    r = ref[t_over[idx], idx]
    # (or, for a reference just past the boundary, a value near it)
    assert np.all((np.isinf(g) | (np.abs(g) >= 0.5 * FMAX[dtype])) & (np.sign(g) == np.sign(r))), \
        f"{name}: out-of-range gradient not an infinity of its sign"


def check_all(w: W.ScanWorkload, inp: dict, layer, ref: dict, lanes=None, widened_frac=1e-3):
    """Every output of a run against the oracle (ref from oracle_expect).
    Returns the counts of elements judged by a widened band (assert_widened
    bounds each by `widened_frac` of its output)."""
    syn = w.neuron == "synaptic"
    counts = check_spikes_and_mem(w, ref, layer.spk, layer.mem, layer.syn if syn else None, lanes)
    rtol, atol = TOL[w.io_dtype]
    gI = lanes_2d(layer.grad_I, lanes)
    over, over_lanes = overflow_mask(ref["grad_I"], w.io_dtype)
    if over_lanes.any():
        check_overflow("grad_I", gI, ref["grad_I"], over, w.io_dtype)
        counts["grad_I_overflow_lanes"] = int(over_lanes.sum())
        print(f"{int(over_lanes.sum())} of {over_lanes.size} lanes' gradients leave the "
              f"{w.io_dtype} range (the float64 BPTT exceeds it)")
    keep = ~over
    counts["grad_I"] = assert_close("grad_I", gI[keep], ref["grad_I"][keep], rtol, atol,
                                    ref["grad_I_scale"][keep])
    f_rtol, f_atol = TOL[W.F32]
    assert np.array_equal(lanes_1d(layer.mem_final, lanes), ref["mem32"][-1]) if w.T > 0 else True
    fine = ~(over_lanes | extreme_lanes(ref["grad_I"]))
    counts["grad_mem0"] = assert_close("grad_mem0", lanes_1d(layer.grad_mem0, lanes)[fine],
                                       ref["grad_mem0"][fine], f_rtol, f_atol,
                                       ref["grad_mem0_scale"][fine])
    if syn:
        counts["grad_syn0"] = assert_close("grad_syn0", lanes_1d(layer.grad_syn0, lanes),
                                           ref["grad_syn0"], f_rtol, f_atol,
                                           ref["grad_syn0_scale"])
    if lanes is None:
        B, N, C, HW = w.B, w.N, w.C, w.HW
        counts["grad_beta"] = check_param_grad("grad_beta", lanes_1d(layer.grad_beta),
                                               ref["grad_beta"], ref["grad_beta_lane"], B, N,
                                               w.beta_mode, C, HW)
        counts["grad_thr"] = check_param_grad("grad_thr", lanes_1d(layer.grad_thr),
                                              ref["grad_thr"], ref["grad_thr_lane"], B, N,
                                              w.thr_mode, C, HW)
        if syn:
            counts["grad_alpha"] = check_param_grad("grad_alpha", lanes_1d(layer.grad_alpha),
                                                    ref["grad_alpha"], ref["grad_alpha_lane"], B,
                                                    N, w.alpha_mode, C, HW)
        if w.neuron == "rleaky":
            counts["grad_v"] = check_param_grad("grad_v", lanes_1d(layer.grad_v), ref["grad_v"],
                                                ref["grad_v_lane"], B, N, w.v_mode, C, HW)
    n_el = ref["spk32"].size
    n_lane = ref["spk32"].shape[1] if ref["spk32"].ndim == 2 else 1
    plen = {"scalar": 1, "per_neuron": w.N, "per_channel": w.C}
    sizes = {"spk_fp64_ambiguous": n_el, "mem_fp32_bound": n_el * (2 if syn else 1),
             "grad_I": n_el, "grad_mem0": n_lane, "grad_syn0": n_lane,
             "grad_beta": plen[w.beta_mode], "grad_thr": plen[w.thr_mode],
             "grad_alpha": plen[w.alpha_mode], "grad_v": plen[w.v_mode]}
    # lanes whose exact gradient leaves the storage range (exploding BPTT)
    # are reported, and bounded separately
    n_over = counts.pop("grad_I_overflow_lanes", 0)
    assert n_over <= 0.05 * n_lane, f"{n_over} of {n_lane} lanes overflow"
    # a parameter with a handful of entries cannot take a fraction: at most
    # one of them may rest on its floor
    for k in ("grad_beta", "grad_thr", "grad_alpha", "grad_v"):
        if k in counts and sizes[k] * widened_frac < 1:
            assert counts[k] <= 1, f"{k}: {counts[k]} of {sizes[k]} judged by the floor"
            counts.pop(k)
    assert_widened(counts, sizes, widened_frac)
    if n_over:
        counts["grad_I_overflow_lanes"] = n_over
    return counts
