"""The paper's convolutional SNN (Tab. I "CSNN": 12C5-MP2-64C5-MP2-10 on
28x28 input) as one training step through the C ABI.  Activations are
channel-last ([T*B, H, W, C] bf16), so every conv layer's Leaky scan runs
over lanes (b, y, x, c) with a per-channel beta (C = channels, one neuron
per channel per run).  Per conv layer:

  im2col -> tensor-core GEMM (the synaptic operation of Fig. 3 over patch
  rows) -> Leaky scan (Eq. 4, reset to zero, learnable per-channel beta)
  -> 2x2 max pool;

then the flattened map feeds a dense Leaky output layer, the rate-coded
cross-entropy (Sec. V-A), BPTT back through every stage (max-pool gradient
to the window's first maximum, scan BPTT with per-channel dL/dbeta, the
GEMM backward and col2im), and AdamW on the weights and the betas.  Only
the sequencing of library calls lives here; every step runs in libsnn's
kernels.

Channel counts are padded to a multiple of 8 (12 -> 16, the 10 outputs ->
16) because the GEMM's TMA tiles need 16-byte row strides.  A padded
channel has zero filters: its current is 0, it never fires, no later
filter reads it, and its gradients are exactly 0.

The first layer (a 5x5 filter over one input channel: 25 products per
output) runs as a direct convolution on the CUDA cores, with its image
staged in shared memory, and so does its weight gradient; a patch-row GEMM
would write and read 32 padded columns per output pixel for that
(``direct_first=False`` keeps the im2col + GEMM path, whose 25 columns are
padded to 32).

``save="fused"`` stores every scan's bf16 membrane trace (the BPTT reads
it instead of recomputing from the currents) and runs the GEMM layers (the
second convolution over its patch rows, the readout) as one kernel each:
the GEMM with the Leaky scan in its epilogue, so their currents never
reach HBM.
"""
from __future__ import annotations

import torch

from . import snn
from . import workloads as W


def _pad8(n: int) -> int:
    return (n + 7) // 8 * 8


class ConvSNN:
    """Buffers and calls of one CSNN training step (forward, loss, BPTT,
    AdamW on the weights and the per-channel betas)."""

    def __init__(self, w: W.ConvWorkload, convs, Wfc, device="cuda", save: str = "recompute",
                 lr: float = 1e-3, betas=(0.9, 0.999), eps: float = 1e-8,
                 weight_decay: float = 1e-2, learn_beta: bool = True,
                 direct_first: bool = True):
        self.w = w
        self.save = save
        self.fused = save == "fused"
        scan_save = "mem" if self.fused else save
        self.lr, self.betas, self.eps, self.weight_decay = lr, betas, eps, weight_decay
        self.learn_beta = learn_beta
        self.batch_total = None
        self.device = torch.device(device)
        dev = self.device
        T, B = w.T, w.B
        self.M = M = T * B
        shapes, n_flat = w.shapes()
        # geometry with padded channels: (H, W, Cin_p, Cout_p, k, Ho, Wo, Hp, Wp, Kpad)
        self.geo = []
        cin_p = w.Cin
        for (h, wd, cin, cout, k, ho, wo, hp, wp) in shapes:
            cout_p = _pad8(cout)
            self.geo.append((h, wd, cin_p, cout_p, k, ho, wo, hp, wp, _pad8(k * k * cin_p)))
            cin_p = cout_p
        hf, wf, cf = self.geo[-1][7], self.geo[-1][8], self.geo[-1][3]
        self.n_flat = hf * wf * cf
        # layers that run as a direct convolution (only the first: it needs
        # no input gradient)
        g0 = self.geo[0]
        self.direct = [direct_first and g0[4] * g0[4] * g0[2] <= 32 and g0[3] <= 16
                       and g0[0] * g0[1] * g0[2] <= 8192] + [False] * (len(self.geo) - 1)
        self.n_out = _pad8(w.n_classes)

        # weights: one flat buffer per quantity, each block on a 64-element
        # boundary, so that one AdamW launch updates every layer
        wshapes = [(g[3], g[9]) for g in self.geo] + [(self.n_out, self.n_flat)]
        offs = [0]
        for r, c in wshapes:
            offs.append(offs[-1] + (r * c + 63) // 64 * 64)
        host = torch.zeros(offs[-1], dtype=torch.bfloat16)
        for l, (Wc, g) in enumerate(zip(convs, self.geo)):
            cout, k, _, cin = Wc.shape
            blk = torch.zeros((g[3], k, k, g[2]), dtype=torch.bfloat16)
            blk[:cout, :, :, :cin] = Wc
            flat = torch.zeros(wshapes[l], dtype=torch.bfloat16)
            flat[:, : k * k * g[2]] = blk.reshape(g[3], -1)
            host[offs[l]: offs[l] + flat.numel()] = flat.reshape(-1)
        cl = shapes[-1][3]
        fc = torch.zeros((self.n_out, hf, wf, cf), dtype=torch.bfloat16)
        fc[: w.n_classes, :, :, :cl] = Wfc.reshape(w.n_classes, hf, wf, cl)
        L = len(self.geo)
        host[offs[L]: offs[L] + fc.numel()] = fc.reshape(-1)
        self.W_flat = host.to(dev)
        self.W32_flat = self.W_flat.float()
        self.m_flat = torch.zeros_like(self.W32_flat)
        self.v_flat = torch.zeros_like(self.W32_flat)
        self.dW_flat = torch.zeros_like(self.W32_flat)
        self.step_counter = torch.zeros(2, dtype=torch.int64, device=dev)

        def view(buf, l):
            r, c = wshapes[l]
            return buf[offs[l]: offs[l] + r * c].view(r, c)

        self.W = [view(self.W_flat, l) for l in range(L + 1)]
        self.dW = [view(self.dW_flat, l) for l in range(L + 1)]

        # per-channel betas of the conv layers: one flat fp32 buffer (its own
        # AdamW state), each layer's block on a 4-element (16-byte) boundary
        boffs = [0]
        for g in self.geo:
            boffs.append(boffs[-1] + (g[3] + 3) // 4 * 4)
        self.beta_flat = torch.full((boffs[-1],), w.beta, dtype=torch.float32, device=dev)
        self.dbeta_flat = torch.zeros_like(self.beta_flat)
        self.bm_flat = torch.zeros_like(self.beta_flat)
        self.bv_flat = torch.zeros_like(self.beta_flat)
        self.beta_counter = torch.zeros(2, dtype=torch.int64, device=dev)
        self.beta = [self.beta_flat[boffs[l]: boffs[l] + g[3]] for l, g in enumerate(self.geo)]
        self.dbeta = [self.dbeta_flat[boffs[l]: boffs[l] + g[3]] for l, g in enumerate(self.geo)]
        self.thr = torch.full((1,), w.thr, dtype=torch.float32, device=dev)
        self.beta_fc = torch.full((1,), w.beta_fc, dtype=torch.float32, device=dev)

        bf = dict(dtype=torch.bfloat16, device=dev)
        self.cols, self.I, self.layers, self.pool, self.idx = [], [], [], [], []
        self.grad_spk, self.grad_pool, self.dcols, self.ws_bwd = [], [], [], []
        for l, (h, wd, cin, cout, k, ho, wo, hp, wp, kpad) in enumerate(self.geo):
            rows = M * ho * wo
            self.cols.append(None if self.direct[l] else torch.empty((rows, kpad), **bf))
            fuse = self.fused and not self.direct[l]  # GEMM and scan in one kernel
            self.I.append(None if fuse else
                          torch.empty((rows, cout), dtype=torch.float32, device=dev))
            lw = W.ScanWorkload(name=f"csnn_conv{l}", neuron="leaky", T=T, B=B,
                                N=ho * wo * cout, C=cout, HW=1, in_dtype=W.F32, io_dtype=W.BF16,
                                beta=("const", w.beta), beta_mode="per_channel",
                                thr=("const", w.thr), reset=w.reset, surrogate="fast_sigmoid",
                                sg_param=w.sg_param, save=scan_save,
                                want_mem=scan_save == "mem")
            self.layers.append(snn.ScanLayer(lw, device=dev))
            self.pool.append(torch.empty((M, hp, wp, cout), **bf))
            self.idx.append(torch.empty((M, hp, wp, cout), dtype=torch.uint8, device=dev))
            self.grad_spk.append(torch.empty((M, ho, wo, cout), **bf))
            self.grad_pool.append(torch.empty((M, hp, wp, cout), **bf))
            self.dcols.append(torch.empty((rows, kpad), **bf) if l > 0 else None)
            if self.direct[l]:
                nb = snn.snn_conv2d_small_dw_workspace_bytes(M, h, wd, cin, cout, k, k)
            else:
                nb = snn.snn_dense_workspace_bytes(rows, kpad, cout)
            self.ws_bwd.append(torch.zeros(max(nb, 256), dtype=torch.uint8, device=dev))
        self.I_fc = None if self.fused else \
            torch.empty((M, self.n_out), dtype=torch.float32, device=dev)
        fw = W.ScanWorkload(name="csnn_out", neuron="leaky", T=T, B=B, N=self.n_out,
                            in_dtype=W.F32, io_dtype=W.BF16, beta=("const", w.beta_fc),
                            thr=("const", w.thr), reset=w.reset, surrogate="fast_sigmoid",
                            sg_param=w.sg_param, save=scan_save, want_mem=scan_save == "mem")
        self.out_layer = snn.ScanLayer(fw, device=dev)
        self.fused_loss = scan_save == "mem"
        self.ws_fwd = torch.zeros(256, dtype=torch.uint8, device=dev)
        self.ws_bwd.append(torch.zeros(snn.snn_dense_workspace_bytes(M, self.n_flat, self.n_out),
                                       dtype=torch.uint8, device=dev))
        self.loss = torch.zeros(1, dtype=torch.float32, device=dev)
        self.ws_loss = torch.zeros(snn.snn_rate_ce_workspace_bytes(B), dtype=torch.uint8,
                                   device=dev)
        self.grad_out = torch.empty((T, B, self.n_out), **bf)

    # -- the step as a list of library calls ---------------------------------

    def layer_input(self, l, X):
        """[T*B, H, W, Cin_p] bf16 input map of conv layer l."""
        return X if l == 0 else self.pool[l - 1]

    def ops(self, X, labels, stream=None, side=None):
        """(name, call) in launch order: per conv layer im2col, GEMM, scan,
        max pool; the output layer's GEMM and scan; the loss; the reverse
        pass from the top; AdamW on the weights and on the betas.  With a
        snn.SideStream the output layer's weight gradient runs on it, beside
        the reverse pass, and the first layer's backward joins it back before
        the update.  The convolutions' weight gradients stay in line: beside
        the second convolution's input-gradient GEMM and the first layer's
        scan they took the SMs those need and the step got longer."""
        T, B, M = self.w.T, self.w.B, self.M
        out = []
        for l, (h, wd, cin, cout, k, ho, wo, hp, wp, kpad) in enumerate(self.geo):
            layer = self.layers[l]
            if self.direct[l]:
                out.append((f"conv_fwd{l}", lambda l=l, k=k, s=(M, ho, wo, cout):
                            snn.snn_conv2d_small_fwd_nhwc(self.layer_input(l, X), self.W[l],
                                                          self.I[l].view(s), k, k, stream)))
            else:
                out.append((f"im2col{l}", lambda l=l, k=k: snn.snn_im2col_nhwc(
                    self.layer_input(l, X), self.cols[l], k, k, stream)))
                if self.I[l] is None:  # fused: the GEMM's epilogue runs the scan
                    out.append((f"conv_scan_fwd{l}", lambda l=l, layer=layer, p=ho * wo:
                                snn.snn_dense_leaky_fwd(layer.desc, self.cols[l], self.W[l],
                                                        self.beta[l], self.thr, layer.spk,
                                                        layer.mem, layer.ckpt, self.ws_fwd, P=p,
                                                        stream=stream)))
                else:
                    out.append((f"conv_fwd{l}", lambda l=l: snn.snn_dense_layer_fwd(
                        self.cols[l], self.W[l], self.I[l], self.ws_fwd, stream)))
            if self.I[l] is not None:
                out.append((f"scan_fwd{l}", lambda l=l, layer=layer: layer.forward(
                    self.I[l].view(T, B, -1), self.beta[l], self.thr, stream=stream)))
            out.append((f"pool_fwd{l}", lambda l=l, layer=layer, s=(M, ho, wo, cout):
                        snn.snn_maxpool2_fwd_nhwc(layer.spk.view(s), self.pool[l], self.idx[l],
                                                  stream)))
        L = len(self.geo)
        flat = self.pool[-1].view(M, -1)
        if self.fused:
            o = self.out_layer
            out.append(("fc_scan_fwd", lambda: snn.snn_dense_leaky_fwd(
                o.desc, flat, self.W[L], self.beta_fc, self.thr, o.spk, o.mem, o.ckpt,
                self.ws_fwd, stream=stream)))
        else:
            out.append(("fc_fwd", lambda: snn.snn_dense_layer_fwd(flat, self.W[L], self.I_fc,
                                                                   self.ws_fwd, stream)))
            out.append(("scan_fwd_out", lambda: self.out_layer.forward(
                self.I_fc.view(T, B, -1), self.beta_fc, self.thr, stream=stream)))
        o = self.out_layer
        if self.fused_loss:  # the readout's trace is stored: its BPTT in the loss launch
            out.append(("ce_loss", lambda: snn.snn_rate_ce_leaky_bwd(
                o.desc, o.spk, labels, self.w.n_classes, self.beta_fc, self.thr, o.mem, None,
                self.loss, self.grad_out, o.grad_I, self.ws_loss, stream,
                batch_total=self.batch_total)))
        else:
            out.append(("ce_loss", lambda: snn.snn_rate_ce_loss(
                o.spk, labels, self.w.n_classes, self.loss, self.grad_out, self.ws_loss, stream,
                batch_total=self.batch_total)))
            out.append(("scan_bwd_out", lambda: o.backward(
                None if self.I_fc is None else self.I_fc.view(T, B, -1), self.beta_fc, self.thr,
                self.grad_out, want_param_grads=False, want_state_grads=False, stream=stream)))
        out.append(("fc_bwd", lambda: snn.dense_layer_bwd_split(
            flat, self.W[L], self.out_layer.grad_I.view(M, -1),
            self.grad_pool[-1].view(M, -1), self.dW[L], self.ws_bwd[L], stream, side)))
        for l in range(L - 1, -1, -1):
            h, wd, cin, cout, k, ho, wo, hp, wp, kpad = self.geo[l]
            layer = self.layers[l]
            out.append((f"pool_bwd{l}", lambda l=l: snn.snn_maxpool2_bwd_nhwc(
                self.grad_pool[l], self.idx[l], self.grad_spk[l], stream)))
            out.append((f"scan_bwd{l}", lambda l=l, layer=layer: self._scan_bwd(l, stream)))
            if self.direct[l]:
                out.append((f"conv_bwd{l}", lambda l=l, layer=layer, k=k, s=(M, ho, wo, cout):
                            snn.snn_conv2d_small_dw_nhwc(self.layer_input(l, X),
                                                         layer.grad_I.view(s), self.dW[l], k, k,
                                                         self.ws_bwd[l], stream)))
            else:
                out.append((f"conv_bwd{l}", lambda l=l, layer=layer, rows=M * ho * wo, c=cout:
                            snn.snn_dense_layer_bwd(self.cols[l], self.W[l],
                                                    layer.grad_I.view(rows, c), self.dcols[l],
                                                    self.dW[l], self.ws_bwd[l], stream)))
            if l == 0 and side is not None:  # the reverse pass ends here
                name, call = out[-1]
                out[-1] = (name, lambda call=call: (call(), side.join(stream)))
            if l > 0:
                out.append((f"col2im{l}", lambda l=l, k=k: snn.snn_col2im_nhwc(
                    self.dcols[l], self.grad_pool[l - 1], k, k, stream)))
        out.append(("adamw", lambda: self.update(stream)))
        return out

    def _scan_bwd(self, l, stream):
        T, B = self.w.T, self.w.B
        layer = self.layers[l]
        recompute = layer.w.save == "recompute"
        I = self.I[l].view(T, B, -1) if recompute else None
        snn.snn_leaky_bwd(layer.desc, I if recompute else None, layer.ckpt, layer.mem, layer.spk,
                          self.beta[l], self.thr, None, self.grad_spk[l].view(T, B, -1), None,
                          None, layer.grad_I, self.dbeta[l], None, None, layer.ws, stream)

    def update(self, stream=None):
        """AdamW on every weight in one launch (rewrites the bf16 copies the
        GEMMs read), then on the betas (no weight decay)."""
        snn.snn_adamw_step(self.W32_flat, self.W_flat, self.dW_flat, self.m_flat, self.v_flat,
                           self.lr, self.betas[0], self.betas[1], self.eps, self.weight_decay,
                           step_counter=self.step_counter, stream=stream)
        if self.learn_beta:
            snn.snn_adamw_step(self.beta_flat, None, self.dbeta_flat, self.bm_flat, self.bv_flat,
                               self.lr, self.betas[0], self.betas[1], self.eps, 0.0,
                               step_counter=self.beta_counter, stream=stream)

    def _n_fwd(self):
        names = [n for n, _ in self.ops(None, None)]
        return names.index("ce_loss") + 1

    def forward(self, X, labels, stream=None):
        """X: bf16 [T*B, H, W, Cin] spikes on the device; labels int32 [B]."""
        for _, call in self.ops(X, labels, stream)[: self._n_fwd()]:
            call()
        return self.loss

    def backward(self, X, stream=None):
        for _, call in self.ops(X, None, stream)[self._n_fwd(): -1]:
            call()
        return self.dW

    def step(self, X, labels, stream=None):
        """Forward, loss and BPTT (parameters unchanged)."""
        self.forward(X, labels, stream)
        return self.backward(X, stream)

    def train_step(self, X, labels, stream=None, side=None):
        """One full training step (weight gradients on `side`, a
        snn.SideStream, if given)."""
        for _, call in self.ops(X, labels, stream, side):
            call()
        return self.loss

    # -- results without padding ---------------------------------------------

    def conv_weight(self, l, buf=None):
        """[Cout, k, k, Cin] filters of conv layer l (fp32 master by default)."""
        h, wd, cin_p, cout_p, k, *_ = self.geo[l]
        cout, _ = self.w.convs[l]
        cin = self.w.Cin if l == 0 else self.w.convs[l - 1][0]
        src = (self.W32_flat if buf is None else buf)
        r, c = cout_p, self.geo[l][9]
        off = self.W[l].storage_offset() - self.W_flat.storage_offset()
        blk = src[off: off + r * c].view(r, c)[:, : k * k * cin_p].reshape(cout_p, k, k, cin_p)
        return blk[:cout, :, :, :cin]

    def fc_weight(self, buf=None):
        """[n_classes, flattened map] readout weights."""
        L = len(self.geo)
        hf, wf, cf = self.geo[-1][7], self.geo[-1][8], self.geo[-1][3]
        cl = self.w.convs[-1][0]
        src = (self.W32_flat if buf is None else buf)
        off = self.W[L].storage_offset() - self.W_flat.storage_offset()
        blk = src[off: off + self.n_out * self.n_flat].view(self.n_out, hf, wf, cf)
        return blk[: self.w.n_classes, :, :, :cl].reshape(self.w.n_classes, -1)
