"""Writes hand_traces.json: small worked examples of the neuron equations,
evaluated in exact rational arithmetic.

The paper prints no worked example with numbers, so these fixtures are the
equations themselves evaluated exactly on small inputs chosen by hand:

* forward traces of Eq. (3) (strict threshold), Eq. (4) (Leaky, reset by
  subtraction), the reset-to-zero and no-reset variants, Eqs. (5)-(6)
  (Synaptic) and Eq. (7) (recurrent Leaky);
* surrogate gradients (Sec. III-B): the derivative of the loss
  L = sum_t gs_t z_t with dz_t/du_t replaced by the fast sigmoid of
  Eqs. (8)-(9), 1 / (1 + k |u_t - thr|)^2, computed here in FORWARD mode
  (one tangent per input and per parameter, carried through the
  recurrence with exact fractions).  The oracle computes the same
  gradients by reverse accumulation, so the two are independent
  derivations of one definition.

With a detached reset, z_{t-1} in the reset term is a constant; the
recurrent term of Eq. (7) is never detached.

Run from the repository root:  python tests/golden/make_golden.py
It imports nothing from this repository.
"""
from __future__ import annotations

import json
import os
from fractions import Fraction as F

HERE = os.path.dirname(os.path.abspath(__file__))
OUT = os.path.join(HERE, "hand_traces.json")


def sg(x: F, k: F) -> F:
    """Fast-sigmoid surrogate dz/du at x = u - thr (Eq. 9 with slope k)."""
    d = 1 + k * abs(x)
    return 1 / (d * d)


def run(neuron: str, I, beta, thr, reset="subtract", alpha=F(0), v=F(0), detach=True,
        gs=None, k=F(1)):
    """Forward trace and, if gs is given, the surrogate gradients of
    L = sum_t gs_t z_t with respect to every I_s and every parameter, each
    by its own forward-mode tangent.

    neuron: "leaky" (Eq. 4, or the reset variants), "synaptic" (Eqs. 5-6,
    the reset acts on u only), "rleaky" (Eq. 7)."""
    T = len(I)
    # tangent seeds: one per input current, then the parameters
    names = [f"I{s}" for s in range(T)] + ["beta", "thr"]
    if neuron == "synaptic":
        names.append("alpha")
    if neuron == "rleaky":
        names.append("v")
    u, i, z = F(0), F(0), 0
    du = {n: F(0) for n in names}  # d u_{t-1} / d n
    di = {n: F(0) for n in names}  # d i_{t-1} / d n
    dz = {n: F(0) for n in names}  # d z_{t-1} / d n (surrogate)
    spk, mem, syn = [], [], []
    grad = {n: F(0) for n in names}
    for t in range(T):
        seed = {n: F(1 if n == f"I{t}" else 0) for n in names}
        # synaptic current (Eq. 5)
        if neuron == "synaptic":
            i_new = alpha * i + I[t]
            di_new = {n: alpha * di[n] + (i if n == "alpha" else 0) + seed[n] for n in names}
            inp, dinp = i_new, di_new
        else:
            i_new, di_new = i, di
            inp, dinp = I[t], seed
        # membrane (Eqs. 4, 6, 7 and the reset variants)
        if neuron == "rleaky":
            un = beta * u + inp + z * (v - thr)
            dun = {}
            for n in names:
                d = beta * du[n] + (u if n == "beta" else 0) + dinp[n]
                d += z * ((1 if n == "v" else 0) - (1 if n == "thr" else 0))
                d += v * dz[n]                       # recurrent path: never detached
                if not detach:
                    d += -thr * dz[n]
                dun[n] = d
        elif reset == "zero":
            keep = 1 - z
            un = beta * keep * u + inp
            dun = {}
            for n in names:
                d = beta * keep * du[n] + (keep * u if n == "beta" else 0) + dinp[n]
                if not detach:
                    d += -beta * u * dz[n]
                dun[n] = d
        else:
            r = thr if reset == "subtract" else F(0)
            un = beta * u + inp - z * r
            dun = {}
            for n in names:
                d = beta * du[n] + (u if n == "beta" else 0) + dinp[n]
                if reset == "subtract":
                    d += -z * (1 if n == "thr" else 0)
                    if not detach:
                        d += -thr * dz[n]
                dun[n] = d
        zn = 1 if un > thr else 0   # Eq. (3), strict
        s = sg(un - thr, k)
        dzn = {n: s * (dun[n] - (1 if n == "thr" else 0)) for n in names}
        if gs is not None:
            for n in names:
                grad[n] += gs[t] * dzn[n]
        u, i, z, du, di, dz = un, i_new, zn, dun, di_new, dzn
        spk.append(zn)
        mem.append(un)
        syn.append(i_new)
    out = {"spk": spk, "mem": mem}
    if neuron == "synaptic":
        out["syn"] = syn
    if gs is not None:
        out["grad_I"] = [grad[f"I{s}"] for s in range(T)]
        for n in names[T:]:
            out[f"grad_{n}"] = grad[n]
    return out


def _q(x) -> str:
    return str(F(x))


def _enc(v):
    if isinstance(v, list):
        return [_enc(e) for e in v]
    if isinstance(v, F):
        return {"exact": _q(v), "value": float(v)}
    return v


I5 = [F(1, 2), F(4, 5), F(3, 10), F(6, 5), F(0)]
I3 = I5[:3]


def cases() -> list:
    """(name, citation, arguments, result) of every fixture."""
    c = []

    def add(name, cite, **kw):
        res = run(**kw)
        args = {k: (_enc(list(v)) if isinstance(v, list) else _enc(v) if isinstance(v, F) else v)
                for k, v in kw.items()}
        c.append({"name": name, "citation": cite, "args": args,
                  "result": {k: _enc(v) for k, v in res.items()}})

    b9, one = F(9, 10), F(1)
    add("leaky_subtract_T5", "Eqs. (3)-(4)", neuron="leaky", I=I5, beta=b9, thr=one)
    add("leaky_zero_reset_T5", "Eq. (3); Eq. (4) with the reset to zero", neuron="leaky", I=I5,
        beta=b9, thr=one, reset="zero")
    add("leaky_no_reset_T5", "Eq. (3); Eq. (4) without the reset term", neuron="leaky", I=I5,
        beta=b9, thr=one, reset="none")
    add("synaptic_subtract_T5", "Eqs. (3), (5)-(6)", neuron="synaptic", I=I5, alpha=F(4, 5),
        beta=b9, thr=one)
    add("tie_at_threshold", "Eq. (3): strict comparison", neuron="leaky", I=[F(1)],
        beta=F(1, 2), thr=one)
    add("rleaky_T5", "Eqs. (3), (7)", neuron="rleaky", I=[F(3, 2), F(1, 5), F(1), F(0), F(9, 10)],
        beta=F(1, 2), thr=one, v=F(1, 4))
    for det in (True, False):
        tag = "detached" if det else "not_detached"
        add(f"bptt_leaky_subtract_T3_{tag}", "Eqs. (3)-(4), (8)-(9); Sec. III-B", neuron="leaky",
            I=I3, beta=b9, thr=one, detach=det, gs=[F(1)] * 3)
        add(f"bptt_leaky_zero_reset_T4_{tag}", "Eqs. (3)-(4) reset to zero, (8)-(9); Sec. III-B",
            neuron="leaky", I=I5[:4], beta=b9, thr=one, reset="zero", detach=det,
            gs=[F(1), F(-1, 2), F(7, 10), F(1)], k=F(2))
        add(f"bptt_synaptic_T4_{tag}", "Eqs. (3), (5)-(6), (8)-(9); Sec. III-B",
            neuron="synaptic", I=I5[:4], alpha=F(4, 5), beta=b9, thr=one, detach=det,
            gs=[F(1), F(1, 2), F(-1, 4), F(1)], k=F(3, 2))
        add(f"bptt_rleaky_T5_{tag}", "Eqs. (3), (7), (8)-(9); Sec. III-B", neuron="rleaky",
            I=[F(3, 2), F(1, 5), F(1), F(0), F(9, 10)], beta=F(1, 2), thr=one, v=F(1, 4),
            detach=det, gs=[F(1), F(-1), F(1, 2), F(1), F(1)])
    return c


def render() -> str:
    return json.dumps({"generator": "tests/golden/make_golden.py", "fixtures": cases()},
                      indent=1) + "\n"


if __name__ == "__main__":
    with open(OUT, "w") as f:
        f.write(render())
    print(f"wrote {OUT}")
