"""The autograd wrapper: gradients through torch's engine equal the C ABI's
own backward, and match the oracle."""
import numpy as np
import pytest
import torch

from paper_2211_10725_gb300 import workloads as W
from paper_2211_10725_gb300.autograd import scan
from tests import scan_harness as H

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("neuron", ["leaky", "synaptic", "rleaky"])
def test_autograd_matches_the_abi_and_the_oracle(neuron, cuda_device):
    w = W.SYNAPTIC_C2.scaled(name=f"ag_{neuron}", neuron=neuron, T=12, B=4, N=256,
                             beta_mode="per_neuron", thr_mode="scalar")
    inp = W.make_scan_inputs(w)
    d = {k: v.to(cuda_device) for k, v in inp.items()}
    third_name = {"synaptic": "alpha", "rleaky": "v"}.get(neuron)
    leaves = {k: d[k].clone().requires_grad_(True) for k in ("I", "beta", "thr")}
    third = d[third_name].clone().requires_grad_(True) if third_name else None
    spk = scan(leaves["I"], leaves["beta"], leaves["thr"], w, third)
    (spk * d["grad_spk"].float()).sum().backward()
    ref_layer = H.run_gpu(w, inp)           # the same step through the C ABI directly
    assert torch.equal(spk.detach(), ref_layer.spk)
    assert torch.equal(leaves["I"].grad, ref_layer.grad_I)
    assert torch.equal(leaves["beta"].grad, ref_layer.grad_beta)
    assert torch.equal(leaves["thr"].grad, ref_layer.grad_thr)
    if third_name:
        got = ref_layer.grad_alpha if neuron == "synaptic" else ref_layer.grad_v
        assert torch.equal(third.grad, got)
    ref = H.oracle_expect(w, inp)
    H.assert_close("grad_I", H.lanes_2d(leaves["I"].grad), ref["grad_I"], *H.TOL[w.io_dtype],
                   ref["grad_I_scale"])
