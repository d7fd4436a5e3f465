"""PyTorch autograd over the C ABI: a scan layer usable inside an ordinary
torch training graph (as snnTorch's neurons are), with the forward and BPTT
running in libsnn's kernels.

``LeakyScan.apply(I, beta, thr, workload)`` returns the spike tensor
[T, B, N]; its backward returns dL/dI and the beta / threshold gradients
(reduced to their layouts).  The Synaptic and recurrent neurons take alpha
or v as a fourth tensor and return its gradient as well.  Only the spike
output is differentiable; the membrane trace is not returned.
"""
from __future__ import annotations

import torch

from . import snn
from . import workloads as W


class _ScanFunction(torch.autograd.Function):
    @staticmethod
    def forward(ctx, I, beta, thr, third, w: W.ScanWorkload):
        layer = snn.ScanLayer(w, device=I.device, want_syn=w.neuron == "synaptic")
        I = I.contiguous()
        kw = {}
        if w.neuron == "synaptic":
            kw["alpha"] = third
        elif w.neuron == "rleaky":
            kw["v"] = third
        layer.forward(I, beta, thr, **kw)
        ctx.layer, ctx.kw = layer, kw
        ctx.save_for_backward(I, beta, thr)
        return layer.spk.clone()

    @staticmethod
    def backward(ctx, grad_spk):
        I, beta, thr = ctx.saved_tensors
        layer = ctx.layer
        g = grad_spk.to(layer.spk.dtype).contiguous()
        layer.backward(I, beta, thr, g, want_state_grads=False, **ctx.kw)
        third = None
        if layer.synaptic:
            third = layer.grad_alpha.clone()
        elif layer.recurrent:
            third = layer.grad_v.clone()
        return layer.grad_I.clone(), layer.grad_beta.clone(), layer.grad_thr.clone(), third, None


def scan(I, beta, thr, w: W.ScanWorkload, third=None):
    """Spikes of a scan layer described by ``w`` (its shape, dtypes, reset,
    surrogate, parameter layouts and save variant); differentiable in I,
    beta, thr and the third parameter (alpha or v)."""
    if (w.T, w.B, w.N) != tuple(I.shape):
        raise ValueError("scan: I does not have the workload's [T, B, N] shape")
    return _ScanFunction.apply(I, beta, thr, third, w)
