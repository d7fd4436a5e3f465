"""The paper's dense SNN (Tab. I "DSNN", here 784-1000-1000-10 Leaky layers)
as one training step through the C ABI: per layer the input current of all
T*B rows in one tensor-core GEMM (the synaptic operation of Fig. 3), then
the fused Leaky scan; the rate-coded cross-entropy loss (Sec. V-A); the
BPTT reverse pass back through every scan and GEMM; and the AdamW update of
the weights (fp32 master copy, bf16 copy for the GEMMs).  Only the
sequencing of library calls lives here; every step runs in libsnn's
kernels.

Layer widths are padded to a multiple of 8 neurons (zero weight rows, so
the 10-neuron output layer has 16) because the GEMM's TMA tiles need row
strides that are multiples of 16 bytes; a padded neuron's current is 0, it
never fires, and its gradients are exactly 0.

The backward recomputes each layer's membrane trace from its input current
and checkpoints (``save="recompute"``) unless ``save="mem"`` asks for the
bf16 trace to be stored by the forward.  ``save="fused"`` stores the trace
too, but runs each layer's forward as one kernel, the GEMM with the Leaky
scan in its epilogue (the currents never reach HBM), and, for T > 1, each
input-gradient product with the BPTT of the layer below in its epilogue (the
spike gradients never reach HBM).  Whenever the readout's trace is stored, the
loss launch also runs the readout's BPTT.
"""
from __future__ import annotations

import torch

from . import snn
from . import workloads as W


def _pad8(n: int) -> int:
    return (n + 7) // 8 * 8


class DenseSNN:
    """Buffers and calls of one DSNN training step (forward, loss, BPTT,
    AdamW update)."""

    def __init__(self, w: W.DenseWorkload, weights, device="cuda", save: str = "recompute",
                 lr: float = 1e-3, betas=(0.9, 0.999), eps: float = 1e-8,
                 weight_decay: float = 1e-2):
        self.w = w
        self.save = save
        self.fused = save == "fused"
        # the input-gradient GEMMs carry the lower layer's BPTT when the scan
        # has a time chain to hide the GEMM behind (T = 1: separate kernels)
        self.fused_bwd = self.fused and w.T > 1
        scan_save = "mem" if self.fused else save
        # with the readout's trace stored, the loss launch also runs its BPTT
        self.fused_loss = scan_save == "mem"
        self.lr, self.betas, self.eps, self.weight_decay = lr, betas, eps, weight_decay
        # batch the loss is averaged over (the global batch under data
        # parallelism; None: this replica's batch)
        self.batch_total = None
        self.device = torch.device(device)
        dev = self.device
        T, B = w.T, w.B
        self.M = T * B
        self.sizes = list(w.sizes)
        self.padded = [self.sizes[0]] + [_pad8(n) for n in self.sizes[1:]]
        # all layers' weights in one flat buffer per quantity (bf16 copy for
        # the GEMMs, fp32 master, AdamW moments, dW), so that one launch
        # updates every layer; each layer's [N_pad, K_pad] block starts on a
        # 64-element boundary
        shapes = [(self.padded[l + 1], self.padded[l]) for l in range(len(weights))]
        offs = [0]
        for n_out, k_in in shapes:
            offs.append(offs[-1] + n_out * k_in)
        host = torch.zeros(offs[-1], dtype=torch.bfloat16)
        for l, Wl in enumerate(weights):
            n_out, k_in = Wl.shape
            host[offs[l]:offs[l + 1]].view(shapes[l])[:n_out, :k_in] = Wl
        self.W_flat = host.to(dev)
        self.W32_flat = self.W_flat.float()
        self.m_flat = torch.zeros_like(self.W32_flat)
        self.v_flat = torch.zeros_like(self.W32_flat)
        self.dW_flat = torch.zeros_like(self.W32_flat)
        self.step_counter = torch.zeros(2, dtype=torch.int64, device=dev)
        self.W = [self.W_flat[offs[l]:offs[l + 1]].view(shapes[l]) for l in range(len(shapes))]
        self.dW = [self.dW_flat[offs[l]:offs[l + 1]].view(shapes[l]) for l in range(len(shapes))]
        self.layers, self.I = [], []
        for l in range(len(weights)):
            n = self.padded[l + 1]
            lw = W.ScanWorkload(name=f"dsnn_layer{l}", neuron="leaky", T=T, B=B, N=n,
                                in_dtype=W.F32, io_dtype=W.BF16, beta=("const", w.beta),
                                thr=("const", w.thr), surrogate="fast_sigmoid",
                                sg_param=w.sg_param, save=scan_save,
                                want_mem=scan_save == "mem")
            self.layers.append(snn.ScanLayer(lw, device=dev))
            self.I.append(None if self.fused else
                          torch.empty((self.M, n), dtype=torch.float32, device=dev))
        self.beta = torch.full((1,), w.beta, dtype=torch.float32, device=dev)
        self.thr = torch.full((1,), w.thr, dtype=torch.float32, device=dev)
        self.ws_fwd = torch.zeros(256, dtype=torch.uint8, device=dev)
        self.ws_bwd = []
        for l in range(len(weights)):
            nb = snn.snn_dense_workspace_bytes(self.M, self.padded[l], self.padded[l + 1])
            self.ws_bwd.append(torch.zeros(nb, dtype=torch.uint8, device=dev))
        self.loss = torch.zeros(1, dtype=torch.float32, device=dev)
        self.ws_loss = torch.zeros(snn.snn_rate_ce_workspace_bytes(B), dtype=torch.uint8,
                                   device=dev)
        self.grad_out = torch.empty((T, B, self.padded[-1]), dtype=torch.bfloat16, device=dev)
        self.grad_in = [torch.empty((self.M, self.padded[l]), dtype=torch.bfloat16, device=dev)
                        for l in range(1, len(weights))]

    def layer_input(self, l, X):
        """[T*B, K] bf16 input of layer l: the data for l = 0, else the spikes
        of layer l - 1."""
        return X if l == 0 else self.layers[l - 1].spk.view(self.M, self.padded[l])

    def _n_fwd(self):
        return (1 if self.fused else 2) * len(self.layers) + 1

    def forward(self, X, labels, stream=None):
        """X: bf16 [T*B, 784] spikes on the device; labels int32 [B]."""
        for _, call in self.ops(X, labels, stream)[: self._n_fwd()]:
            call()
        return self.loss

    def backward(self, X, stream=None):
        """BPTT from the loss gradient of the last forward; returns dW."""
        for _, call in self.ops(X, None, stream)[self._n_fwd(): -1]:
            call()
        return self.dW

    def update(self, stream=None):
        """AdamW on every layer in one launch; rewrites the bf16 weights the
        GEMMs read.  The step number lives on the device (graph-replayable)."""
        snn.snn_adamw_step(self.W32_flat, self.W_flat, self.dW_flat, self.m_flat, self.v_flat,
                           self.lr, self.betas[0], self.betas[1], self.eps, self.weight_decay,
                           step_counter=self.step_counter, stream=stream)

    def ops(self, X, labels, stream=None, side=None):
        """The training step as a list of (name, call) in launch order: per
        layer the forward GEMM and scan, the loss, per layer from the top the
        scan BPTT and the dense backward, then the AdamW update.  With a
        snn.SideStream the weight gradients of the upper layers run on it,
        beside the input-gradient products of the reverse pass, and the last
        dense backward joins it back before the update."""
        T, B = self.w.T, self.w.B
        out = []
        for l, layer in enumerate(self.layers):
            if self.fused:
                out.append((f"dense_scan_fwd{l}", lambda l=l, layer=layer: snn.snn_dense_leaky_fwd(
                    layer.desc, self.layer_input(l, X), self.W[l], self.beta, self.thr,
                    layer.spk, layer.mem, layer.ckpt, self.ws_fwd, stream=stream)))
                continue
            out.append((f"dense_fwd{l}", lambda l=l: snn.snn_dense_layer_fwd(
                self.layer_input(l, X), self.W[l], self.I[l], self.ws_fwd, stream)))
            out.append((f"scan_fwd{l}", lambda l=l, layer=layer: layer.forward(
                self.I[l].view(T, B, -1), self.beta, self.thr, stream=stream)))
        top = len(self.layers) - 1
        o = self.layers[top]
        if self.fused_loss:
            out.append(("ce_loss", lambda: snn.snn_rate_ce_leaky_bwd(
                o.desc, o.spk, labels, self.w.n_classes, self.beta, self.thr, o.mem, None,
                self.loss, self.grad_out, o.grad_I, self.ws_loss, stream,
                batch_total=self.batch_total, pop=self.w.pop)))
        else:
            out.append(("ce_loss", lambda: snn.snn_rate_ce_loss(
                o.spk, labels, self.w.n_classes, self.loss, self.grad_out, self.ws_loss, stream,
                batch_total=self.batch_total, pop=self.w.pop)))
        for l in range(top, -1, -1):
            grad = self.grad_out if l == top else self.grad_in[l].view(T, B, -1)
            if (l == top and not self.fused_loss) or (l < top and not self.fused_bwd):
                out.append((f"scan_bwd{l}", lambda l=l, grad=grad: self.layers[l].backward(
                    None if self.I[l] is None else self.I[l].view(T, B, -1), self.beta,
                    self.thr, grad, want_param_grads=False, want_state_grads=False,
                    stream=stream)))
            # fused: layer l's input gradient is the spike gradient of layer
            # l - 1, whose BPTT runs in the epilogue of that product
            dX = self.grad_in[l - 1] if (l > 0 and not self.fused_bwd) else None
            out.append((f"dense_bwd{l}", lambda l=l, dX=dX: self._dense_bwd(
                l, X, dX, stream, side)))
            if l > 0 and self.fused_bwd:
                lo = self.layers[l - 1]
                out.append((f"dense_scan_bwd{l}", lambda l=l, lo=lo: snn.snn_dense_leaky_bwd(
                    lo.desc, self.layers[l].grad_I.view(self.M, -1), self.W[l], self.beta,
                    self.thr, lo.mem, lo.spk, lo.ckpt, lo.grad_I, self.ws_fwd, stream)))
        out.append(("adamw", lambda: self.update(stream)))
        return out

    def _dense_bwd(self, l, X, dX, stream, side):
        dI = self.layers[l].grad_I.view(self.M, -1)
        if side is not None and l == 0:
            # the last product of the reverse pass: on the main stream, then
            # wait for the weight gradients forked onto the side stream
            snn.snn_dense_layer_bwd(self.layer_input(l, X), self.W[l], dI, dX, self.dW[l],
                                    self.ws_bwd[l], stream)
            side.join(stream)
            return
        snn.dense_layer_bwd_split(self.layer_input(l, X), self.W[l], dI, dX, self.dW[l],
                                  self.ws_bwd[l], stream, side)

    def step(self, X, labels, stream=None):
        """Forward, loss and BPTT (weights unchanged); returns the dW list."""
        self.forward(X, labels, stream)
        return self.backward(X, stream)

    def train_step(self, X, labels, stream=None, side=None):
        """One full training step: forward, loss, BPTT and the AdamW update
        (the upper layers' weight gradients on `side`, a snn.SideStream, if
        given)."""
        for _, call in self.ops(X, labels, stream, side):
            call()
        return self.loss

    def weight_grads(self):
        """dW of each layer without the padding rows/columns."""
        return [self.dW[l][: self.sizes[l + 1], : self.sizes[l]] for l in range(len(self.dW))]
