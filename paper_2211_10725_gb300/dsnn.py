"""The paper's dense SNN (Tab. I "DSNN", here 784-1000-1000-10 Leaky layers)
as one training step through the C ABI: per layer the input current of all
T*B rows in one tensor-core GEMM (the synaptic operation of Fig. 3), then
the fused Leaky scan; the rate-coded cross-entropy loss (Sec. V-A); and the
BPTT reverse pass back through every scan and GEMM.  Only the sequencing of
library calls lives here; every step runs in libsnn's kernels.

Layer widths are padded to a multiple of 8 neurons (zero weight rows, so
the 10-neuron output layer has 16) because the GEMM's TMA tiles need row
strides that are multiples of 16 bytes; a padded neuron's current is 0, it
never fires, and its gradients are exactly 0.

The backward recomputes each layer's membrane trace from its input current
and checkpoints (``save="recompute"``) unless ``save="mem"`` asks for the
bf16 trace to be stored by the forward.
"""
from __future__ import annotations

import torch

from . import snn
from . import workloads as W


def _pad8(n: int) -> int:
    return (n + 7) // 8 * 8


class DenseSNN:
    """Buffers and calls of one DSNN training step (forward, loss, BPTT)."""

    def __init__(self, w: W.DenseWorkload, weights, device="cuda", save: str = "recompute"):
        self.w = w
        self.save = save
        self.device = torch.device(device)
        dev = self.device
        T, B = w.T, w.B
        self.M = T * B
        self.sizes = list(w.sizes)
        self.padded = [self.sizes[0]] + [_pad8(n) for n in self.sizes[1:]]
        self.W = []
        for l, Wl in enumerate(weights):
            n_out, k_in = Wl.shape
            Wp = torch.zeros((self.padded[l + 1], self.padded[l]), dtype=torch.bfloat16)
            Wp[:n_out, :k_in] = Wl
            self.W.append(Wp.to(dev))
        self.layers, self.I = [], []
        for l in range(len(weights)):
            n = self.padded[l + 1]
            lw = W.ScanWorkload(name=f"dsnn_layer{l}", neuron="leaky", T=T, B=B, N=n,
                                in_dtype=W.F32, io_dtype=W.BF16, beta=("const", w.beta),
                                thr=("const", w.thr), surrogate="fast_sigmoid",
                                sg_param=w.sg_param, save=save, want_mem=save == "mem")
            self.layers.append(snn.ScanLayer(lw, device=dev))
            self.I.append(torch.empty((self.M, n), dtype=torch.float32, device=dev))
        self.beta = torch.full((1,), w.beta, dtype=torch.float32, device=dev)
        self.thr = torch.full((1,), w.thr, dtype=torch.float32, device=dev)
        self.ws_fwd = torch.zeros(256, dtype=torch.uint8, device=dev)
        self.ws_bwd = []
        for l in range(len(weights)):
            nb = snn.snn_dense_workspace_bytes(self.M, self.padded[l], self.padded[l + 1])
            self.ws_bwd.append(torch.zeros(nb, dtype=torch.uint8, device=dev))
        self.loss = torch.zeros(1, dtype=torch.float32, device=dev)
        self.grad_out = torch.empty((T, B, self.padded[-1]), dtype=torch.bfloat16, device=dev)
        self.grad_in = [torch.empty((self.M, self.padded[l]), dtype=torch.bfloat16, device=dev)
                        for l in range(1, len(weights))]
        self.dW = [torch.empty((self.padded[l + 1], self.padded[l]), dtype=torch.float32,
                               device=dev) for l in range(len(weights))]

    def layer_input(self, l, X):
        """[T*B, K] bf16 input of layer l: the data for l = 0, else the spikes
        of layer l - 1."""
        return X if l == 0 else self.layers[l - 1].spk.view(self.M, self.padded[l])

    def forward(self, X, labels, stream=None):
        """X: bf16 [T*B, 784] spikes on the device; labels int32 [B]."""
        for l, layer in enumerate(self.layers):
            snn.snn_dense_layer_fwd(self.layer_input(l, X), self.W[l], self.I[l], self.ws_fwd,
                                    stream)
            layer.forward(self.I[l].view(self.w.T, self.w.B, -1), self.beta, self.thr,
                          stream=stream)
        snn.snn_rate_ce_loss(self.layers[-1].spk, labels, self.sizes[-1], self.loss,
                             self.grad_out, stream)
        return self.loss

    def backward(self, X, stream=None):
        grad = self.grad_out
        for l in range(len(self.layers) - 1, -1, -1):
            layer = self.layers[l]
            layer.backward(self.I[l].view(self.w.T, self.w.B, -1), self.beta, self.thr, grad,
                           want_param_grads=False, want_state_grads=False, stream=stream)
            dX = self.grad_in[l - 1] if l > 0 else None
            snn.snn_dense_layer_bwd(self.layer_input(l, X), self.W[l],
                                    layer.grad_I.view(self.M, -1), dX, self.dW[l],
                                    self.ws_bwd[l], stream)
            if l > 0:
                grad = dX.view(self.w.T, self.w.B, -1)
        return self.dW

    def step(self, X, labels, stream=None):
        self.forward(X, labels, stream)
        return self.backward(X, stream)

    def weight_grads(self):
        """dW of each layer without the padding rows/columns."""
        return [self.dW[l][: self.sizes[l + 1], : self.sizes[l]] for l in range(len(self.dW))]
