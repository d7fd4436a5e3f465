"""The oracle against the worked examples in tests/golden/hand_traces.json:
the neuron equations (Eqs. 3-7) and their surrogate gradients (Eqs. 8-9,
Sec. III-B) evaluated in exact rational arithmetic, the gradients in forward
mode, by tests/golden/make_golden.py (which imports nothing from this
repository).  The oracle's float64 forward must give the same spikes and
states, and its reverse-mode BPTT the same gradients."""
import json
import os
import sys

import numpy as np
import pytest

from oracle import snn_oracle as O

HERE = os.path.dirname(os.path.abspath(__file__))
GOLDEN = os.path.join(HERE, "golden", "hand_traces.json")
sys.path.insert(0, os.path.join(HERE, "golden"))
import make_golden  # noqa: E402

FIXTURES = json.load(open(GOLDEN))["fixtures"]


def test_fixture_file_is_what_the_generator_writes():
    with open(GOLDEN) as f:
        assert f.read() == make_golden.render()


def _val(x):
    if isinstance(x, list):
        return np.array([_val(e) for e in x], dtype=np.float64)
    if isinstance(x, dict):
        return x["value"]
    return x


@pytest.mark.parametrize("fx", FIXTURES, ids=[f["name"] for f in FIXTURES])
def test_oracle_matches_exact_worked_example(fx):
    a = fx["args"]
    r = fx["result"]
    I = _val(a["I"])[:, None]
    beta, thr = [_val(a["beta"])], [_val(a["thr"])]
    reset = a.get("reset", "subtract")
    neuron = a["neuron"]
    if neuron == "leaky":
        spk, mem = O.leaky_forward(I, beta, thr, reset)
        syn = None
    elif neuron == "synaptic":
        spk, mem, syn = O.synaptic_forward(I, [_val(a["alpha"])], beta, thr, reset)
    else:
        spk, mem = O.rleaky_forward(I, [_val(a["v"])], beta, thr)
        syn = None
    assert spk[:, 0].tolist() == r["spk"]
    np.testing.assert_allclose(mem[:, 0], _val(r["mem"]), rtol=1e-13, atol=1e-14)
    if syn is not None:
        np.testing.assert_allclose(syn[:, 0], _val(r["syn"]), rtol=1e-13, atol=1e-14)
    if "gs" not in a:
        return
    gs = _val(a["gs"])[:, None]
    kw = dict(detach=a["detach"], sg="fast_sigmoid", sg_param=_val(a["k"]) if "k" in a else 1.0)
    if neuron == "leaky":
        g = O.leaky_backward(mem, spk, gs, beta, thr, reset, **kw)
    elif neuron == "synaptic":
        g = O.synaptic_backward(mem, spk, syn, gs, [_val(a["alpha"])], beta, thr, reset, **kw)
    else:
        g = O.rleaky_backward(mem, spk, gs, [_val(a["v"])], beta, thr, **kw)
    np.testing.assert_allclose(g["grad_I"][:, 0], _val(r["grad_I"]), rtol=1e-11, atol=1e-13)
    for name, key in [("grad_beta", "grad_beta_lane"), ("grad_thr", "grad_thr_lane"),
                      ("grad_alpha", "grad_alpha_lane"), ("grad_v", "grad_v_lane")]:
        if name in r:
            np.testing.assert_allclose(g[key][0], _val(r[name]), rtol=1e-11, atol=1e-13)
