"""The dense layer with its Leaky scan in the GEMM epilogue
(snn_dense_leaky_fwd) against the oracle's GEMM followed by its Leaky
forward, and the dense SNN step built on it.

Comparison protocol: the layer inputs are 0/1 spikes and the weights bf16
values flushed to zero below 2^-7 in magnitude (and at most 0.25).  Every
product is then a multiple of 2^-14 and every partial sum of at most 1024
of them stays below 2^8, so each current is exact in fp32 whatever the
summation order.  The fused kernel's fp32 trace must then equal the
oracle's float32 Leaky forward bit for bit: spikes, the bf16-rounded
membrane and the spike bits.
"""
import ctypes

import numpy as np
import pytest
import torch

from oracle import snn_oracle as O
from paper_2211_10725_gb300 import snn
from paper_2211_10725_gb300 import workloads as W

pytestmark = pytest.mark.gpu

# T, B, P, K, Nout, reset, parameter mode
CASES = [
    (25, 16, 1, 784, 128, "subtract", "scalar"),
    (25, 128, 1, 784, 1000, "subtract", "scalar"),     # the 784-1000 layer at full size
    (25, 128, 1, 1000, 16, "subtract", "scalar"),      # the padded 10-neuron readout
    (1, 128, 1, 3072, 1000, "subtract", "scalar"),     # the population network, T = 1
    (3, 7, 1, 64, 40, "zero", "per_neuron"),
    (128, 3, 1, 32, 24, "none", "per_neuron"),          # one row per tile
    (25, 4, 64, 400, 64, "zero", "per_channel"),       # a convolution's patch rows
    (5, 3, 9, 16, 8, "subtract", "per_channel"),
    (7, 19, 1, 200, 136, "zero", "scalar"),            # ragged tiles in both dimensions
]


def _np(t):
    return t.detach().to("cpu", torch.float32).numpy().astype(np.float64)


def _unpack_bits(ckpt, T, L):
    row = ((L + 7) // 8 + 15) // 16 * 16
    raw = ckpt.cpu().view(torch.uint8).numpy()[: T * row].reshape(T, row)[:, : (L + 7) // 8]
    return np.unpackbits(raw, axis=1, bitorder="little")[:, :L].astype(np.float64)


def _exact_weights(shape, g):
    w = ((torch.rand(shape, generator=g) * 2 - 1) * 0.25).to(torch.bfloat16)
    w[w.float().abs() < 2.0 ** -7] = 0
    return w


@pytest.mark.parametrize("T,B,P,K,Nout,reset,mode", CASES)
def test_fused_forward_matches_oracle(T, B, P, K, Nout, reset, mode, cuda_device):
    g = torch.Generator().manual_seed(T * 1000 + B * 10 + K + Nout)
    R = B * P
    X = (torch.rand((T, R, K), generator=g) < 0.2).to(torch.bfloat16)
    Wt = _exact_weights((Nout, K), g)
    per = mode != "scalar"
    beta = (0.8 + 0.19 * torch.rand(Nout if per else 1, generator=g)).float()
    thr = (0.7 + 0.6 * torch.rand(Nout if per else 1, generator=g)).float()
    w = W.ScanWorkload(name="fused", neuron="leaky", T=T, B=B, N=P * Nout, C=Nout, HW=1,
                       in_dtype=W.F32, io_dtype=W.BF16, beta_mode=mode, thr_mode=mode,
                       reset=reset, save="mem", want_mem=True)
    desc = snn.make_desc(w)
    L = B * P * Nout
    spk = torch.empty((T, B, P * Nout), dtype=torch.bfloat16, device=cuda_device)
    mem = torch.empty_like(spk)
    ckpt = torch.zeros(snn.snn_scan_ckpt_elems(desc, False), dtype=torch.float32,
                       device=cuda_device)
    ws = torch.zeros(256, dtype=torch.uint8, device=cuda_device)
    snn.snn_dense_leaky_fwd(desc, X.reshape(T * R, K).to(cuda_device), Wt.to(cuda_device),
                            beta.to(cuda_device), thr.to(cuda_device), spk, mem, ckpt, ws, P=P)
    torch.cuda.synchronize()
    assert snn.snn_workspace_status(ws) == 0
    # oracle: the currents, then the Leaky forward in float32
    I = (_np(X).reshape(T * R, K) @ _np(Wt).T).reshape(T, L)
    assert np.array_equal(I.astype(np.float32).astype(np.float64), I)  # exact sums
    lanes_b = O.lane_param(beta.numpy(), B, P * Nout, mode, Nout, 1)
    lanes_t = O.lane_param(thr.numpy(), B, P * Nout, mode, Nout, 1)
    s_ref, m_ref = O.leaky_forward(I.astype(np.float32), lanes_b.astype(np.float32),
                                   lanes_t.astype(np.float32), reset, dtype=np.float32)
    got_s = _np(spk).reshape(T, L)
    assert np.array_equal(got_s, s_ref.astype(np.float64)), "spikes"
    assert np.array_equal(_np(mem).reshape(T, L), O.bf16_round(m_ref.astype(np.float64))), "mem"
    assert np.array_equal(_unpack_bits(ckpt, T, L), got_s), "spike bits"
    assert 0 < got_s.mean() < 1


def test_fused_argument_checks(cuda_device):
    w = W.ScanWorkload(name="fused", neuron="leaky", T=4, B=2, N=16, in_dtype=W.F32,
                       io_dtype=W.BF16, save="mem", want_mem=True)
    buf = torch.zeros(1 << 16, dtype=torch.float32, device=cuda_device)
    X = buf[:4 * 2 * 16].view(8, 16).to(torch.bfloat16)
    Wt = torch.zeros((16, 16), dtype=torch.bfloat16, device=cuda_device)
    p = torch.ones(1, device=cuda_device)
    spk = torch.empty((4, 2, 16), dtype=torch.bfloat16, device=cuda_device)
    ws = torch.zeros(256, dtype=torch.uint8, device=cuda_device)
    lib = snn.load_library()

    def call(desc, P=1, K=16, x=X, mem=spk):
        return lib.snn_dense_leaky_fwd(ctypes.byref(desc), P, K, x.data_ptr(), Wt.data_ptr(),
                                       p.data_ptr(), p.data_ptr(), spk.data_ptr(), mem.data_ptr(),
                                       None, ws.data_ptr(), 256, None)

    assert call(snn.make_desc(w)) == 0
    assert call(snn.make_desc(w.scaled(save="recompute"))) == 3       # needs the stored trace
    assert call(snn.make_desc(w.scaled(io_dtype=W.F32))) == 3
    assert call(snn.make_desc(w.scaled(T=129))) == 3
    assert call(snn.make_desc(w), K=12) == 3                           # K % 8
    assert call(snn.make_desc(w), P=3) == 1                            # N % P
    assert call(snn.make_desc(w.scaled(N=12))) == 3                    # Nout % 8
    assert call(snn.make_desc(w), x=buf[1:].view(-1)[:128].view(8, 16)) == 2  # alignment
    torch.cuda.synchronize()
