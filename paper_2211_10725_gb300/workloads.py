"""Seeded synthetic workloads for the spiking-neuron scan.

This module only draws random inputs and describes workload shapes: it holds
none of the neuron arithmetic, so both the CUDA path and the CPU oracle can be
fed from it.  Every tensor is drawn on the CPU with ``torch.Generator`` so that
the same seed gives the same values on any machine.

Workloads (all synthetic; MNIST/CIFAR-10 shapes from the paper's Tab. I stand
in for the datasets, which are not used):

* ``leaky_T25_B128_N1000``      Leaky LIF layer (Eq. 4), fp32.
* ``synaptic_T100_B128_N4096``  current-based LIF layer (Eqs. 5-6), fp32.
* ``dsnn_784_1000_1000_10``     3-layer dense SNN, bf16 GEMMs, T=25, B=128.
* ``dsnn_pop_3072_1000_500_T1``  2-layer dense SNN with a population-coded
                                output (50 neurons per class), T=1.
* ``conv_lif_T25_B128``         LIF on the conv-SNN activation shapes
                                [12,24,24] and [64,8,8], per-channel beta.
* ``leaky_bf16_T500_B64_N8192`` large Leaky layer, bf16 storage, per-neuron
                                beta/threshold.
* ``rleaky_T25_B128_N1000``     recurrent Leaky layer (Eq. 7), fp32, per-neuron v.
* ``rleaky_bf16_T500_B64_N8192`` large recurrent Leaky layer, bf16 storage.
* ``csnn_12c5_mp2_64c5_mp2_10_T25_B128`` convolutional SNN on 28x28 input
                                (Tab. I CSNN), per-channel learnable beta.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import torch

SEED_BASE = 2211_10725

F32, BF16, F16 = "f32", "bf16", "f16"
TORCH_DTYPE = {F32: torch.float32, BF16: torch.bfloat16, F16: torch.float16}


@dataclasses.dataclass(frozen=True)
class ScanWorkload:
    """Shape and distribution of one scan layer's synthetic inputs."""

    name: str
    neuron: str                 # "leaky" (Eq. 4), "synaptic" (Eqs. 5-6), "rleaky" (Eq. 7)
    T: int
    B: int
    N: int                      # flattened neurons per sample (C*H*W for conv maps)
    C: int = 1                  # channels (per-channel parameters)
    HW: int = 1                 # spatial size per channel
    in_dtype: str = F32         # dtype of the input current I
    io_dtype: str = F32         # dtype of spk, mem, grad_spk, grad_I
    i_mean: float = 0.3
    i_std: float = 0.5          # second argument of N(mu, s) is the std deviation
    beta: tuple = ("const", 0.9)        # ("const", v) | ("uniform", lo, hi)
    thr: tuple = ("const", 1.0)
    alpha: tuple = ("const", 0.8)
    beta_mode: str = "scalar"   # scalar | per_neuron | per_channel
    thr_mode: str = "scalar"
    alpha_mode: str = "scalar"
    v: tuple = ("uniform", -0.5, 0.5)   # recurrent weight (rleaky)
    v_mode: str = "per_neuron"
    reset: str = "subtract"     # subtract | zero | none
    surrogate: str = "fast_sigmoid"     # fast_sigmoid | atan
    sg_param: float = 25.0
    detach_reset: bool = True
    save: str = "mem"           # mem | recompute
    ckpt_every: int = 8
    want_mem: bool = True       # the layer's mem output is requested
    seed_index: int = 0

    def scaled(self, **kw) -> "ScanWorkload":
        return dataclasses.replace(self, **kw)

    @property
    def lanes(self) -> int:
        return self.B * self.N

    @property
    def neuron_steps(self) -> int:
        return self.T * self.B * self.N


LEAKY_C1 = ScanWorkload(
    name="leaky_T25_B128_N1000", neuron="leaky", T=25, B=128, N=1000,
    i_mean=0.3, i_std=0.5, surrogate="fast_sigmoid", sg_param=25.0, seed_index=0)

SYNAPTIC_C2 = ScanWorkload(
    name="synaptic_T100_B128_N4096", neuron="synaptic", T=100, B=128, N=4096,
    i_mean=0.2, i_std=0.4, alpha=("const", 0.8), surrogate="atan", sg_param=2.0,
    seed_index=1)

CONV_C4A = ScanWorkload(
    name="conv_lif_T25_B128_C12x24x24", neuron="leaky", T=25, B=128, N=12 * 24 * 24,
    C=12, HW=24 * 24, i_mean=0.25, i_std=0.5, beta=("const", 0.95),
    beta_mode="per_channel", reset="zero", surrogate="fast_sigmoid", sg_param=25.0,
    want_mem=False, seed_index=3)

CONV_C4B = CONV_C4A.scaled(name="conv_lif_T25_B128_C64x8x8", N=64 * 8 * 8, C=64, HW=64)

BIG_C5 = ScanWorkload(
    name="leaky_bf16_T500_B64_N8192", neuron="leaky", T=500, B=64, N=8192,
    in_dtype=BF16, io_dtype=BF16, i_mean=0.1, i_std=0.3,
    beta=("uniform", 0.85, 0.99), thr=("uniform", 0.8, 1.2),
    beta_mode="per_neuron", thr_mode="per_neuron", surrogate="atan", sg_param=2.0,
    save="recompute", ckpt_every=8, want_mem=False, seed_index=4)

# Recurrent Leaky neuron (Eq. 7; the paper's recurrent SNN of Fig. 6a): the
# C1 and C5 shapes with a one-to-one recurrent weight v ~ U(-0.5, 0.5) per
# neuron.
RLEAKY_C6 = LEAKY_C1.scaled(name="rleaky_T25_B128_N1000", neuron="rleaky", seed_index=6)
RLEAKY_C7 = BIG_C5.scaled(name="rleaky_bf16_T500_B64_N8192", neuron="rleaky", seed_index=7)

SCAN_WORKLOADS = {w.name: w for w in (LEAKY_C1, SYNAPTIC_C2, CONV_C4A, CONV_C4B, BIG_C5,
                                      RLEAKY_C6, RLEAKY_C7)}


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    return g


def _param(spec: tuple, mode: str, w: ScanWorkload, g: torch.Generator) -> torch.Tensor:
    n = {"scalar": 1, "per_neuron": w.N, "per_channel": w.C}[mode]
    if spec[0] == "const":
        return torch.full((n,), float(spec[1]), dtype=torch.float32)
    if spec[0] == "uniform":
        lo, hi = spec[1], spec[2]
        return (lo + (hi - lo) * torch.rand(n, generator=g, dtype=torch.float32))
    raise ValueError(spec)


def make_scan_inputs(w: ScanWorkload, seed: Optional[int] = None,
                     with_mem0: bool = False, with_grad_mem: bool = False,
                     with_grad_final: bool = False) -> dict:
    """Draw the layer's inputs on the CPU.

    Returns a dict of CPU tensors: ``I`` [T,B,N] in_dtype, ``grad_spk`` [T,B,N]
    io_dtype ~ N(0,1), ``beta``/``thr``/``alpha`` fp32 of length 1, N or C, and
    optionally ``mem0``/``syn0`` [B,N] fp32, ``grad_mem`` [T,B,N] io_dtype and
    ``grad_mem_final``/``grad_syn_final`` [B,N] fp32; ``v`` (length 1, N or
    C) for the recurrent neuron.
    """
    seed = SEED_BASE + w.seed_index if seed is None else seed
    g = _gen(seed)
    shape = (w.T, w.B, w.N)
    I = (w.i_mean + w.i_std * torch.randn(shape, generator=g, dtype=torch.float32))
    out = {"I": I.to(TORCH_DTYPE[w.in_dtype])}
    out["beta"] = _param(w.beta, w.beta_mode, w, g)
    out["thr"] = _param(w.thr, w.thr_mode, w, g)
    if w.neuron == "synaptic":
        out["alpha"] = _param(w.alpha, w.alpha_mode, w, g)
    if w.neuron == "rleaky":
        out["v"] = _param(w.v, w.v_mode, w, g)
    out["grad_spk"] = torch.randn(shape, generator=g, dtype=torch.float32).to(
        TORCH_DTYPE[w.io_dtype])
    if with_mem0:
        out["mem0"] = 0.5 * torch.randn((w.B, w.N), generator=g, dtype=torch.float32) + 0.5
        if w.neuron == "synaptic":
            out["syn0"] = 0.3 * torch.randn((w.B, w.N), generator=g, dtype=torch.float32)
    if with_grad_mem:
        out["grad_mem"] = (0.1 * torch.randn(shape, generator=g, dtype=torch.float32)).to(
            TORCH_DTYPE[w.io_dtype])
    if with_grad_final:
        out["grad_mem_final"] = torch.randn((w.B, w.N), generator=g, dtype=torch.float32)
        if w.neuron == "synaptic":
            out["grad_syn_final"] = torch.randn((w.B, w.N), generator=g, dtype=torch.float32)
    return out


# ---------------------------------------------------------------------------
# 3-layer dense SNN (784-1000-1000-10, T=25, B=128)
# ---------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class DenseWorkload:
    name: str = "dsnn_784_1000_1000_10_T25_B128"
    T: int = 25
    B: int = 128
    sizes: tuple = (784, 1000, 1000, 10)
    rate_max: float = 0.3
    beta: float = 0.9
    thr: float = 1.0
    sg_param: float = 25.0      # fast-sigmoid slope
    n_classes: int = 10
    pop: int = 1                # output neurons per class (population code, Sec. VII)
    seed_index: int = 2

    def scaled(self, **kw) -> "DenseWorkload":
        return dataclasses.replace(self, **kw)


DSNN_C3 = DenseWorkload()

# Population-coded output (Sec. VII): one time step, a CIFAR-10-sized input
# (32x32x3, synthetic spikes as for C3), 50 output neurons per class.
DSNN_POP = DenseWorkload(name="dsnn_pop_3072_1000_500_T1_B128", T=1, B=128,
                         sizes=(3072, 1000, 500), pop=50, seed_index=8)

DENSE_WORKLOADS = {w.name: w for w in (DSNN_C3, DSNN_POP)}


def make_dense_inputs(w: DenseWorkload, seed: Optional[int] = None) -> dict:
    """Bernoulli input spikes with a per-(sample, pixel) rate ~ U(0, rate_max)
    drawn once and independent over t; He-uniform bf16 weights without bias;
    uniform labels in 0..n_classes-1."""
    seed = SEED_BASE + w.seed_index if seed is None else seed
    g = _gen(seed)
    k0 = w.sizes[0]
    rate = w.rate_max * torch.rand((w.B, k0), generator=g, dtype=torch.float32)
    u = torch.rand((w.T, w.B, k0), generator=g, dtype=torch.float32)
    X = (u < rate.unsqueeze(0)).to(torch.bfloat16)
    Ws = []
    for fan_in, fan_out in zip(w.sizes[:-1], w.sizes[1:]):
        bound = (6.0 / fan_in) ** 0.5
        Wl = (2.0 * torch.rand((fan_out, fan_in), generator=g, dtype=torch.float32) - 1.0) * bound
        Ws.append(Wl.to(torch.bfloat16))
    labels = torch.randint(0, w.n_classes, (w.B,), generator=g, dtype=torch.int64).to(torch.int32)
    return {"X": X, "W": Ws, "labels": labels}


# ---------------------------------------------------------------------------
# Convolutional SNN (Tab. I CSNN: 12C5-MP2-64C5-MP2-10 on 28x28, T=25, B=128)
# ---------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class ConvWorkload:
    name: str = "csnn_12c5_mp2_64c5_mp2_10_T25_B128"
    T: int = 25
    B: int = 128
    H: int = 28
    W: int = 28
    Cin: int = 1
    convs: tuple = ((12, 5), (64, 5))   # (output channels, square kernel) per layer
    n_classes: int = 10
    rate_max: float = 0.3
    beta: float = 0.95          # initial per-channel beta of the conv layers
    beta_fc: float = 0.95       # output layer's beta (scalar, fixed)
    thr: float = 1.0
    sg_param: float = 25.0      # fast-sigmoid slope
    reset: str = "zero"
    seed_index: int = 9

    def scaled(self, **kw) -> "ConvWorkload":
        return dataclasses.replace(self, **kw)

    def shapes(self):
        """Per conv layer (H, W, Cin, Cout, k, Ho, Wo, Hp, Wp); then the
        flattened size of the last pooled map."""
        out, h, wd, c = [], self.H, self.W, self.Cin
        for cout, k in self.convs:
            ho, wo = h - k + 1, wd - k + 1
            out.append((h, wd, c, cout, k, ho, wo, ho // 2, wo // 2))
            h, wd, c = ho // 2, wo // 2, cout
        return out, h * wd * c


CSNN_C4 = ConvWorkload()

CONV_WORKLOADS = {w.name: w for w in (CSNN_C4,)}


def make_conv_inputs(w: ConvWorkload, seed: Optional[int] = None) -> dict:
    """Bernoulli input spikes [T, B, H, W, Cin] (channel-last) with a
    per-(sample, pixel) rate ~ U(0, rate_max) drawn once and independent over
    t; He-uniform bf16 filters [Cout, k, k, Cin] and readout weights [10,
    flattened pooled map (y, x, c order)] without bias; uniform labels."""
    seed = SEED_BASE + w.seed_index if seed is None else seed
    g = _gen(seed)
    rate = w.rate_max * torch.rand((w.B, w.H, w.W, w.Cin), generator=g, dtype=torch.float32)
    u = torch.rand((w.T, w.B, w.H, w.W, w.Cin), generator=g, dtype=torch.float32)
    X = (u < rate.unsqueeze(0)).to(torch.bfloat16)
    layers, n_flat = w.shapes()
    convs = []
    for (_, _, cin, cout, k, *_rest) in layers:
        bound = (6.0 / (k * k * cin)) ** 0.5
        Wc = (2.0 * torch.rand((cout, k, k, cin), generator=g, dtype=torch.float32) - 1.0) * bound
        convs.append(Wc.to(torch.bfloat16))
    bound = (6.0 / n_flat) ** 0.5
    Wfc = (2.0 * torch.rand((w.n_classes, n_flat), generator=g, dtype=torch.float32) - 1.0) * bound
    labels = torch.randint(0, w.n_classes, (w.B,), generator=g, dtype=torch.int64).to(torch.int32)
    return {"X": X, "convs": convs, "Wfc": Wfc.to(torch.bfloat16), "labels": labels}
