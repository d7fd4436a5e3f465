"""The dense layer with its Leaky scan in the GEMM epilogue
(snn_dense_leaky_fwd) against the oracle's GEMM followed by its Leaky
forward; the input-gradient GEMM with the lower layer's BPTT in its
epilogue (snn_dense_leaky_bwd) against the oracle's product followed by its
Leaky backward; the rate-coded loss with the readout's BPTT in the same
launch (snn_rate_ce_leaky_bwd) against the oracle's loss and Leaky backward.

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


# The fused backward (snn_dense_leaky_bwd): the spike gradient of the lower
# layer is dI_up @ W computed on the tensor cores and never stored; its BPTT
# runs on the stored bf16 trace.  dI_up is k/16 (|k| <= 16) and W is k/1024
# (|k| < 256): every product is a multiple of 2^-14 and every partial sum of
# at most 1024 of them stays below 2^8, so the spike gradient is exact in fp32
# and the oracle's float64 BPTT on the same stored state is the reference,
# within the bf16 storage tolerance of grad_I.
# T, B, K (upper neurons), N (lower neurons), reset, parameter mode, surrogate,
# detached reset, spike source
BWD_CASES = [
    (25, 16, 128, 64, "subtract", "scalar", "fast_sigmoid", True, "bits"),
    (25, 128, 1000, 1000, "subtract", "scalar", "fast_sigmoid", True, "bits"),  # DSNN 1000-1000
    (25, 128, 16, 1000, "subtract", "scalar", "fast_sigmoid", True, "bits"),    # under the readout
    (1, 128, 1000, 3072, "subtract", "scalar", "fast_sigmoid", True, "bits"),   # T = 1
    (3, 7, 40, 64, "zero", "per_neuron", "atan", False, "spk"),
    (128, 3, 24, 32, "none", "per_neuron", "fast_sigmoid", True, "bits"),       # one row per tile
    (7, 19, 136, 200, "subtract", "scalar", "atan", False, "bits"),             # ragged tiles
    (5, 33, 64, 328, "zero", "scalar", "fast_sigmoid", False, "spk"),
]


def _pack_bits(z, T, L):
    """Spike bits as the store-mode BPTT reads them (bit k of byte j of row t
    is z_t of lane 8j + k; rows padded to 16 bytes)."""
    row = ((L + 7) // 8 + 15) // 16 * 16
    out = np.zeros((T, row), dtype=np.uint8)
    out[:, : (L + 7) // 8] = np.packbits(z.astype(np.uint8), axis=1, bitorder="little")
    return torch.from_numpy(out.reshape(-1)).view(torch.float32)


@pytest.mark.parametrize("T,B,K,N,reset,mode,sg,detach,src", BWD_CASES)
def test_fused_backward_matches_oracle(T, B, K, N, reset, mode, sg, detach, src, cuda_device):
    g = torch.Generator().manual_seed(7 * T + 13 * B + K + 3 * N)
    L = B * N
    dI_up = (torch.randint(-16, 17, (T * B, K), generator=g).float() / 16).to(torch.bfloat16)
    Wt = (torch.randint(-255, 256, (K, N), generator=g).float() / 1024).to(torch.bfloat16)
    per = mode != "scalar"
    beta = (0.8 + 0.19 * torch.rand(N if per else 1, generator=g)).float()
    thr = (0.7 + 0.6 * torch.rand(N if per else 1, generator=g)).float()
    # a stored trace near the threshold and spikes mostly consistent with it
    mem = (torch.randn((T, B, N), generator=g) * 0.6 + 0.9).to(torch.bfloat16)
    lanes_t = O.lane_param(thr.numpy(), B, N, mode, N, 1)
    lanes_b = O.lane_param(beta.numpy(), B, N, mode, N, 1)
    z = (_np(mem).reshape(T, L) > lanes_t[None, :]).astype(np.float64)
    flip = torch.rand((T, L), generator=g).numpy() < 0.02
    z[flip] = 1 - z[flip]
    w = W.ScanWorkload(name="fused_bwd", neuron="leaky", T=T, B=B, N=N, C=N, HW=1,
                       in_dtype=W.F32, io_dtype=W.BF16, beta_mode=mode, thr_mode=mode,
                       reset=reset, surrogate=sg, sg_param=25.0 if sg == "fast_sigmoid" else 2.0,
                       detach_reset=detach, save="mem", want_mem=True)
    desc = snn.make_desc(w)
    spk = torch.from_numpy(z.reshape(T, B, N)).to(torch.bfloat16)
    ckpt = _pack_bits(z, T, L).to(cuda_device) if src == "bits" else None
    gI = torch.full((T, B, N), float("nan"), dtype=torch.bfloat16, device=cuda_device)
    ws = torch.zeros(256, dtype=torch.uint8, device=cuda_device)
    snn.snn_dense_leaky_bwd(desc, dI_up.to(cuda_device), Wt.to(cuda_device), beta.to(cuda_device),
                            thr.to(cuda_device), mem.to(cuda_device),
                            spk.to(cuda_device) if src == "spk" else None, ckpt, gI, ws)
    torch.cuda.synchronize()
    assert snn.snn_workspace_status(ws) == 0
    gs = (_np(dI_up) @ _np(Wt)).reshape(T, L)
    assert np.array_equal(gs.astype(np.float32).astype(np.float64), gs)  # exact sums
    kw = dict(reset=reset, detach=detach, sg=sg, sg_param=w.sg_param)
    ref = O.leaky_backward(_np(mem).reshape(T, L), z, gs, lanes_b, lanes_t, **kw)["grad_I"]
    scale = np.maximum(np.abs(ref), O.leaky_backward(_np(mem).reshape(T, L), z, np.abs(gs),
                                                     lanes_b, lanes_t, **kw)["grad_I"])
    got = _np(gI).reshape(T, L)
    assert np.isfinite(got).all()
    lim = 1e-3 + 2e-2 * scale
    bad = np.abs(got - ref) > lim
    assert not bad.any(), f"{bad.sum()} of {bad.size} beyond tolerance"
    assert np.abs(ref).max() > 0


def test_fused_backward_argument_checks(cuda_device):
    w = W.ScanWorkload(name="fused_bwd", neuron="leaky", T=4, B=2, N=16, in_dtype=W.F32,
                       io_dtype=W.BF16, save="mem", want_mem=True)
    buf = torch.zeros(1 << 16, dtype=torch.float32, device=cuda_device)
    dI = buf[:8 * 16].view(8, 16).to(torch.bfloat16)
    Wt = torch.zeros((16, 16), dtype=torch.bfloat16, device=cuda_device)
    p = torch.ones(1, device=cuda_device)
    mem = torch.zeros((4, 2, 16), dtype=torch.bfloat16, device=cuda_device)
    gI = torch.empty_like(mem)
    ws = torch.zeros(256, dtype=torch.uint8, device=cuda_device)
    lib = snn.load_library()

    def call(desc, K=16, spk=mem, ckpt=None, dI_up=dI):
        return lib.snn_dense_leaky_bwd(ctypes.byref(desc), K, dI_up.data_ptr(), Wt.data_ptr(),
                                       p.data_ptr(), p.data_ptr(), mem.data_ptr(),
                                       None if spk is None else spk.data_ptr(),
                                       None if ckpt is None else ckpt.data_ptr(),
                                       gI.data_ptr(), ws.data_ptr(), 256, None)

    assert call(snn.make_desc(w)) == 0
    assert call(snn.make_desc(w), spk=None) == 1                        # no spike source
    assert call(snn.make_desc(w.scaled(save="recompute"))) == 3
    assert call(snn.make_desc(w.scaled(io_dtype=W.F32))) == 3
    assert call(snn.make_desc(w.scaled(T=129))) == 3
    assert call(snn.make_desc(w), K=12) == 3                            # K % 8
    assert call(snn.make_desc(w.scaled(N=12))) == 3                     # N % 8
    assert call(snn.make_desc(w.scaled(beta_mode="per_channel", C=4, HW=4))) == 3
    assert call(snn.make_desc(w), dI_up=buf[1:].view(-1)[:128].view(8, 16)) == 2  # alignment
    torch.cuda.synchronize()


# The rate-coded loss with the readout's BPTT in the same launch
# (snn_rate_ce_leaky_bwd) against the oracle's loss followed by its Leaky
# backward on the same stored state.
# T, B, C, pop, ld, reset, parameter mode, surrogate, detached reset, io dtype, spike source
CE_CASES = [
    (25, 128, 10, 1, 16, "subtract", "scalar", "fast_sigmoid", True, torch.bfloat16, "spk"),
    (25, 128, 10, 1, 16, "subtract", "scalar", "fast_sigmoid", True, torch.bfloat16, "bits"),
    (1, 128, 10, 50, 504, "subtract", "scalar", "fast_sigmoid", True, torch.bfloat16, "spk"),
    (7, 37, 13, 7, 96, "zero", "per_neuron", "atan", False, torch.float32, "spk"),
    (30, 5, 3, 1, 8, "none", "per_neuron", "fast_sigmoid", False, torch.bfloat16, "bits"),
    (9, 300, 100, 1, 104, "subtract", "scalar", "atan", False, torch.float32, "bits"),
]


@pytest.mark.parametrize("T,B,C,pop,ld,reset,mode,sg,detach,dtype,src", CE_CASES)
def test_rate_ce_with_readout_bptt(T, B, C, pop, ld, reset, mode, sg, detach, dtype, src,
                                   cuda_device):
    g = torch.Generator().manual_seed(T + 3 * B + C + ld)
    L = B * ld
    spk = (torch.rand((T, B, ld), generator=g) < 0.3).to(dtype)
    spk[:, :, C * pop:] = 0
    mem = (torch.randn((T, B, ld), generator=g) * 0.6 + 0.9).to(dtype)
    labels = torch.randint(0, C, (B,), generator=g, dtype=torch.int32)
    per = mode != "scalar"
    beta = (0.8 + 0.19 * torch.rand(ld if per else 1, generator=g)).float()
    thr = (0.7 + 0.6 * torch.rand(ld if per else 1, generator=g)).float()
    w = W.ScanWorkload(name="readout", neuron="leaky", T=T, B=B, N=ld, C=ld, HW=1,
                       in_dtype=W.F32, io_dtype=W.BF16 if dtype == torch.bfloat16 else W.F32,
                       beta_mode=mode, thr_mode=mode, reset=reset, surrogate=sg,
                       sg_param=25.0 if sg == "fast_sigmoid" else 2.0, detach_reset=detach,
                       save="mem", want_mem=True)
    z = _np(spk).reshape(T, L)
    d = lambda t: t.to(cuda_device)
    ckpt = d(_pack_bits(z, T, L)) if src == "bits" else None
    loss = torch.zeros(1, dtype=torch.float32, device=cuda_device)
    gs = torch.full((T, B, ld), float("nan"), dtype=dtype, device=cuda_device)
    gI = torch.full((T, B, ld), float("nan"), dtype=dtype, device=cuda_device)
    ws = torch.zeros(snn.snn_rate_ce_workspace_bytes(B), dtype=torch.uint8, device=cuda_device)
    spk_in = d(spk)
    if src == "bits":   # the spike decisions must come from the bits: spk keeps the counts only
        assert np.array_equal(_np(spk_in.cpu()).reshape(T, L), z)
    snn.snn_rate_ce_leaky_bwd(snn.make_desc(w), spk_in, d(labels), C, d(beta), d(thr), d(mem),
                              ckpt, loss, gs, gI, ws, pop=pop)
    torch.cuda.synchronize()
    rl, rg = O.rate_ce_loss(_np(spk[:, :, :C * pop]), labels.numpy(), pop)
    assert abs(loss.item() - rl) <= 1e-6 * max(1.0, abs(rl))
    full = np.zeros((T, B, ld))
    full[:, :, :C * pop] = rg
    got_gs = _np(gs.cpu())
    assert np.all(got_gs[:, :, C * pop:] == 0)
    rtol = 1e-5 if dtype == torch.float32 else 2e-2
    np.testing.assert_allclose(got_gs, full, rtol=rtol, atol=1e-7 * np.abs(rg).max())
    lanes_b = O.lane_param(beta.numpy(), B, ld, mode, ld, 1)
    lanes_t = O.lane_param(thr.numpy(), B, ld, mode, ld, 1)
    kw = dict(reset=reset, detach=detach, sg=sg, sg_param=w.sg_param)
    m = _np(mem).reshape(T, L)
    ref = O.leaky_backward(m, z, full.reshape(T, L), lanes_b, lanes_t, **kw)["grad_I"]
    scale = np.maximum(np.abs(ref), O.leaky_backward(m, z, np.abs(full.reshape(T, L)), lanes_b,
                                                     lanes_t, **kw)["grad_I"])
    got = _np(gI.cpu()).reshape(T, L)
    assert np.isfinite(got).all()
    floor = (1e-6 if dtype == torch.float32 else 1e-3) * np.abs(ref).max()
    bad = np.abs(got - ref) > floor + rtol * scale
    assert not bad.any(), f"{bad.sum()} of {bad.size} beyond tolerance"
    assert np.abs(ref).max() > 0


def test_rate_ce_with_readout_bptt_argument_checks(cuda_device):
    T, B, C, ld = 4, 2, 3, 8
    w = W.ScanWorkload(name="readout", neuron="leaky", T=T, B=B, N=ld, in_dtype=W.F32,
                       io_dtype=W.BF16, save="mem", want_mem=True)
    buf = torch.zeros(1 << 12, dtype=torch.float32, device=cuda_device)
    p = torch.ones(1, device=cuda_device)
    lab = torch.zeros(B, dtype=torch.int32, device=cuda_device)
    out = torch.zeros(1, dtype=torch.float32, device=cuda_device)   # the loss
    ws = torch.zeros(snn.snn_rate_ce_workspace_bytes(B), dtype=torch.uint8, device=cuda_device)
    lib = snn.load_library()
    x = buf.data_ptr()

    def call(desc, C=C, pop=1, total=0, spk=x, nbytes=None):
        return lib.snn_rate_ce_leaky_bwd(ctypes.byref(desc), C, pop, total, spk, lab.data_ptr(),
                                         p.data_ptr(), p.data_ptr(), x + 1024, None, out.data_ptr(),
                                         x + 2048, x + 3072, ws.data_ptr(),
                                         ws.numel() if nbytes is None else nbytes, None)

    assert call(snn.make_desc(w)) == 0
    assert call(snn.make_desc(w), C=5, pop=2) == 1                      # C*pop > ld
    assert call(snn.make_desc(w), total=1) == 1                        # batch_total < B
    assert call(snn.make_desc(w.scaled(save="recompute"))) == 3        # needs the stored trace
    assert call(snn.make_desc(w.scaled(beta_mode="per_channel", C=2, HW=4))) == 3
    assert call(snn.make_desc(w), spk=x + 2) == 2                       # alignment
    assert call(snn.make_desc(w), nbytes=64) == 4                       # workspace
    torch.cuda.synchronize()
