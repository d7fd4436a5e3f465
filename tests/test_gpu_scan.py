"""Parity of the CUDA scan (through the C ABI) with the CPU oracle.

Small cases sweep every mode (neuron, reset, detach, surrogate, parameter
layout, save variant, dtype pair, optional inputs) over shapes that span
several CTAs with a ragged last strip and shapes whose rows are not 16-byte
multiples (the plain per-lane kernels).  Full-size cases run each workload
in the launch configuration the benchmark times.
"""
import numpy as np
import pytest
import torch

from paper_2211_10725_gb300 import snn
from paper_2211_10725_gb300 import workloads as W
from tests import scan_harness as H
from oracle import snn_oracle as O

pytestmark = pytest.mark.gpu

SHAPES = [(1, 1, 7), (2, 3, 5), (5, 2, 64), (33, 5, 1000), (17, 4, 2048), (9, 3, 1368)]
CHANNELS = {7: (7, 1), 5: (5, 1), 64: (4, 16), 1000: (10, 100), 2048: (8, 256), 1368: (6, 228)}
DTYPES = [(W.F32, W.F32), (W.BF16, W.BF16), (W.F16, W.F16), (W.F32, W.BF16)]
RESETS = ["subtract", "zero", "none"]
MODES = ["scalar", "per_neuron", "per_channel"]


def small_case(i):
    T, B, N = SHAPES[i % len(SHAPES)]
    C, HW = CHANNELS[N]
    in_dt, io_dt = DTYPES[(i // 5) % len(DTYPES)]
    save = ["mem", "recompute"][(i // 3) % 2]
    w = W.ScanWorkload(
        name=f"small{i}", neuron=["leaky", "synaptic"][(i // 11) % 2], T=T, B=B, N=N, C=C, HW=HW,
        in_dtype=in_dt, io_dtype=io_dt, i_mean=0.5, i_std=0.6,
        beta=("uniform", 0.5, 0.95), thr=("uniform", 0.6, 1.4), alpha=("uniform", 0.3, 0.9),
        beta_mode=MODES[(i // 7) % 3], thr_mode=MODES[(i // 2) % 3], alpha_mode=MODES[i % 3],
        reset=RESETS[i % 3], detach_reset=(i % 2 == 0),
        surrogate=["fast_sigmoid", "atan"][(i // 2) % 2], sg_param=[25.0, 2.0][(i // 2) % 2],
        save=save, ckpt_every=[1, 3, 4, 8][(i // 4) % 4], want_mem=True, seed_index=100 + i)
    opts = dict(with_mem0=(i % 4 == 0), with_grad_mem=(i % 5 == 1), with_grad_final=(i % 3 == 0))
    return w, opts


@pytest.mark.parametrize("i", range(72))
def test_small_cases(i, cuda_device):
    w, opts = small_case(i)
    inp = W.make_scan_inputs(w, **opts)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    H.check_all(w, inp, layer, H.oracle_expect(w, inp))


@pytest.mark.parametrize("i", [3, 4, 15, 16, 27, 28, 40, 51, 63])
def test_staged_and_plain_kernels_agree(i, cuda_device):
    w, opts = small_case(i)
    inp = W.make_scan_inputs(w, **opts)
    a = H.run_gpu(w, inp)
    b = H.run_gpu(w, inp, debug_flags=snn.DEBUG_FORCE_PLAIN)
    assert torch.equal(a.spk, b.spk) and torch.equal(a.mem, b.mem)
    assert torch.equal(a.mem_final, b.mem_final)
    if w.save == "recompute" and a.ckpt is not None:
        assert torch.equal(a.ckpt, b.ckpt)
    # the reverse passes accumulate in different orders (packed FMAs vs
    # scalar): they agree within the fp32 gradient tolerance
    H.assert_close("grad_I", H.lanes_2d(a.grad_I), H.lanes_2d(b.grad_I), *H.TOL[w.io_dtype])


def _unpack_bits(ckpt, T, L):
    """Spike bits (bit k of byte j of row t = lane 8j + k; rows padded to 16
    bytes) as a [T, L] 0/1 array."""
    row = ((L + 7) // 8 + 15) // 16 * 16
    raw = ckpt.cpu().view(torch.uint8).numpy()[: T * row].reshape(T, row)[:, : (L + 7) // 8]
    return np.unpackbits(raw, axis=1, bitorder="little")[:, :L].astype(np.float64)


@pytest.mark.parametrize("neuron", ["leaky", "synaptic"])
@pytest.mark.parametrize("io", [W.BF16, W.F16])
@pytest.mark.parametrize("T,B,N", [(9, 3, 1368), (4, 7, 1000), (3, 1, 8)])
def test_store_mode_spike_bits(neuron, io, T, B, N, cuda_device):
    """Store mode with half io: the forward's spike bits equal spk, and the
    backward from the bits (spk not passed) equals the backward from spk."""
    w = W.ScanWorkload(name="bits", neuron=neuron, T=T, B=B, N=N, in_dtype=io, io_dtype=io,
                       save="mem", surrogate="atan", sg_param=2.0, reset="zero",
                       beta=("uniform", 0.5, 0.95), thr=("uniform", 0.6, 1.4), i_mean=0.5,
                       beta_mode="per_neuron", seed_index=7)
    inp = W.make_scan_inputs(w)
    d = {k: v.to(cuda_device) for k, v in inp.items()}
    layer = snn.ScanLayer(w, device=cuda_device, want_syn=True)
    assert layer.ckpt is not None      # the bit rows
    layer.forward(d["I"], d["beta"], d["thr"], d.get("alpha"))
    torch.cuda.synchronize()
    bits = _unpack_bits(layer.ckpt, T, B * N)
    assert np.array_equal(bits, H.lanes_2d(layer.spk))
    spk = layer.spk
    layer.spk = None                   # the backward must not need it
    try:
        layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], alpha=d.get("alpha"))
    finally:
        layer.spk = spk
    g_bits = layer.grad_I.clone()
    gb_bits = layer.grad_beta.clone()
    ckpt = layer.ckpt
    layer.ckpt = None                  # now from the spk rows
    layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], alpha=d.get("alpha"))
    layer.ckpt = ckpt
    torch.cuda.synchronize()
    assert layer.status() == 0
    assert torch.equal(g_bits, layer.grad_I)
    assert torch.equal(gb_bits, layer.grad_beta)
    H.check_all(w, inp, layer, H.oracle_expect(w, inp))


def test_store_mode_without_spk_or_bits_is_rejected(cuda_device):
    w = W.LEAKY_C1.scaled(io_dtype=W.BF16, in_dtype=W.BF16, T=3, B=2, N=16)
    layer = snn.ScanLayer(w, device=cuda_device)
    inp = {k: v.to(cuda_device) for k, v in W.make_scan_inputs(w).items()}
    layer.forward(inp["I"], inp["beta"], inp["thr"])
    layer.spk, layer.ckpt = None, None
    with pytest.raises(snn.SnnError):
        layer.backward(inp["I"], inp["beta"], inp["thr"], inp["grad_spk"])


def test_backward_is_deterministic(cuda_device):
    w = W.SYNAPTIC_C2.scaled(T=20, B=16)
    inp = W.make_scan_inputs(w)
    a = H.run_gpu(w, inp)
    g1 = (a.grad_beta.clone(), a.grad_thr.clone(), a.grad_I.clone())
    a.backward(*[v.cuda() for v in (inp["I"], inp["beta"], inp["thr"], inp["grad_spk"])],
               alpha=inp["alpha"].cuda())
    torch.cuda.synchronize()
    assert torch.equal(g1[0], a.grad_beta) and torch.equal(g1[1], a.grad_thr)
    assert torch.equal(g1[2], a.grad_I)


def test_empty_inputs(cuda_device):
    # B = 0: nothing to scan; parameter gradients are zero-filled
    w = W.LEAKY_C1.scaled(B=0)
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp)
    assert float(layer.grad_beta.abs().sum()) == 0.0
    # T = 0: final state is the initial state, grad_mem0 is grad_mem_final
    w = W.LEAKY_C1.scaled(T=0, B=2, N=64)
    inp = W.make_scan_inputs(w, with_mem0=True, with_grad_final=True)
    layer = H.run_gpu(w, inp)
    assert torch.equal(layer.mem_final.cpu(), inp["mem0"])
    assert torch.equal(layer.grad_mem0.cpu(), inp["grad_mem_final"])
    assert float(layer.grad_beta.abs().sum()) == 0.0


def test_wait_timeout_reports_status_and_context_survives(cuda_device):
    # the producer issues nothing, so the consumers' bounded wait runs out
    w = W.LEAKY_C1.scaled(T=8, B=4, N=1024)
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp, debug_flags=snn.DEBUG_PRODUCER_IDLE, wait_limit_ns=2_000_000)
    assert layer.status() == 6          # SNN_ERR_TIMEOUT, read and cleared
    assert layer.status() == 0
    ok = H.run_gpu(w, inp)
    assert ok.status() == 0
    H.check_all(w, inp, ok, H.oracle_expect(w, inp))


@pytest.mark.parametrize("T,B,N,C", [(5, 3, 9216, 16), (4, 7, 4096, 64), (3, 5, 48, 16),
                                     (6, 2, 8, 2), (2, 1, 256, 256), (25, 128, 9216, 16)])
@pytest.mark.parametrize("neuron", ["leaky", "synaptic"])
def test_channel_last_parameter_gradients(T, B, N, C, neuron, cuda_device):
    """Per-channel parameters on channel-last lanes (one position per
    channel run, the channel of lane l is l % C, as in a convolutional
    layer's [H, W, C] map): the coalesced reduction path, up to the CSNN's
    first-layer shape."""
    w = W.ScanWorkload(name=f"chlast_{neuron}_{T}_{B}_{N}_{C}", neuron=neuron, T=T, B=B, N=N, C=C,
                       HW=1, i_mean=0.5, i_std=0.6, beta=("uniform", 0.5, 0.95),
                       thr=("uniform", 0.6, 1.4), alpha=("uniform", 0.3, 0.9),
                       beta_mode="per_channel", thr_mode="per_channel", alpha_mode="per_channel",
                       reset="zero", save="recompute", want_mem=True, seed_index=400 + C + T)
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    H.check_all(w, inp, layer, H.oracle_expect(w, inp))
    again = H.run_gpu(w, inp)
    assert torch.equal(layer.grad_beta, again.grad_beta)   # fixed summation order


# ---------------------------------------------------------------------------
# Full-size workloads
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("name", ["leaky_T25_B128_N1000", "synaptic_T100_B128_N4096",
                                  "conv_lif_T25_B128_C12x24x24", "conv_lif_T25_B128_C64x8x8"])
def test_full_size_workloads(name, cuda_device):
    w = W.SCAN_WORKLOADS[name]
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    H.check_all(w, inp, layer, H.oracle_expect(w, inp))


def check_every_lane_in_blocks(w, inp, layer, block=1024):
    """Compare a [T, B, N] workload with the oracle on every lane, in blocks
    of `block` neurons with all B samples of each (so per-neuron parameter
    gradients are exact sums of the block's lanes).  Returns the summed
    widened-band counts."""
    host = H.HostCopy(layer)
    totals = {}
    for n0 in range(0, w.N, block):
        ns = np.arange(n0, min(w.N, n0 + block))
        lanes = (np.arange(w.B)[:, None] * w.N + ns[None, :]).reshape(-1)
        ref = H.oracle_expect(w, inp, lanes=lanes)
        for k, v in H.check_all(w, inp, host, ref, lanes=lanes).items():
            totals[k] = totals.get(k, 0) + v
        pnames = ["beta", "thr"] + (["v"] if w.neuron == "rleaky" else [])
        # neurons with a lane whose gradient leaves the storage range have no
        # representable parameter gradient
        # neurons with a lane whose gradients approach the fp32 range have no
        # fp32 parameter gradient (its per-lane sums can overflow part-way)
        _, over = H.overflow_mask(ref["grad_I"], w.io_dtype)
        bad = over | H.extreme_lanes(ref["grad_I"])
        fine = ~bad.reshape(w.B, len(ns)).any(axis=0)
        for pname in pnames:
            part = ref[f"grad_{pname}_lane"].reshape(w.B, len(ns))[:, fine]
            got = H.lanes_1d(getattr(host, f"grad_{pname}"))[ns][fine]
            H.assert_close(f"grad_{pname}", got, part.sum(0), 1e-5,
                           1e-5 * np.abs(part).sum(0) + 1e-6)
    print(w.name, w.save, "widened-band counts over all lanes:", totals)
    return totals


@pytest.mark.parametrize("save,k", [("recompute", 16), ("recompute", 12), ("recompute", 8),
                                    ("mem", 8)])
def test_full_size_large_bf16(save, k, cuda_device):
    """T=500, B=64, N=8192, bf16 storage (the benchmark's workload, in the
    launch configuration it times): every one of the 524,288 lanes against
    the oracle."""
    w = W.BIG_C5.scaled(save=save, ckpt_every=k)
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    check_every_lane_in_blocks(w, inp, layer)


@pytest.mark.parametrize("neuron,dt,save", [("leaky", W.F32, "mem"), ("synaptic", W.F32, "mem"),
                                            ("leaky", W.BF16, "recompute"),
                                            ("synaptic", W.F16, "recompute")])
def test_ring_wraps_with_many_warps(neuron, dt, save, cuda_device):
    # T well beyond the ring depth and strips of hundreds of lanes per CTA, so
    # every stage is refilled many times while a dozen consumer warps read it
    w = W.SYNAPTIC_C2.scaled(name="wrap", neuron=neuron, T=120, B=64, N=4096, in_dtype=dt,
                             io_dtype=dt, save=save, ckpt_every=8)
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    rng = np.random.default_rng(9)
    lanes = np.sort(rng.choice(w.B * w.N, 20000, replace=False))
    H.check_all(w, inp, layer, H.oracle_expect(w, inp, lanes=lanes), lanes=lanes)


# ---------------------------------------------------------------------------
# Recurrent Leaky neuron (Eq. 7)
# ---------------------------------------------------------------------------

def rleaky_case(i):
    T, B, N = SHAPES[i % len(SHAPES)]
    C, HW = CHANNELS[N]
    in_dt, io_dt = DTYPES[(i // 3) % len(DTYPES)]
    w = W.ScanWorkload(
        name=f"rleaky{i}", neuron="rleaky", T=T, B=B, N=N, C=C, HW=HW, in_dtype=in_dt,
        io_dtype=io_dt, i_mean=0.5, i_std=0.6, beta=("uniform", 0.5, 0.95),
        thr=("uniform", 0.6, 1.4), v=("uniform", -0.6, 0.6),
        beta_mode=MODES[(i // 5) % 3], thr_mode=MODES[(i // 2) % 3], v_mode=MODES[i % 3],
        detach_reset=(i % 2 == 0), surrogate=["fast_sigmoid", "atan"][(i // 4) % 2],
        sg_param=[25.0, 2.0][(i // 4) % 2], save=["mem", "recompute"][(i // 6) % 2],
        ckpt_every=[8, 3][(i // 12) % 2], want_mem=True, seed_index=300 + i)
    opts = dict(with_mem0=(i % 4 == 1), with_grad_mem=(i % 5 == 2), with_grad_final=(i % 3 == 1))
    return w, opts


@pytest.mark.parametrize("i", range(24))
def test_rleaky_small_cases(i, cuda_device):
    w, opts = rleaky_case(i)
    inp = W.make_scan_inputs(w, **opts)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    H.check_all(w, inp, layer, H.oracle_expect(w, inp))


@pytest.mark.parametrize("i", [2, 3, 8, 9, 15, 20])
def test_rleaky_staged_and_plain_kernels_agree(i, cuda_device):
    w, opts = rleaky_case(i)
    inp = W.make_scan_inputs(w, **opts)
    a = H.run_gpu(w, inp)
    b = H.run_gpu(w, inp, debug_flags=snn.DEBUG_FORCE_PLAIN)
    assert torch.equal(a.spk, b.spk) and torch.equal(a.mem, b.mem)
    assert torch.equal(a.mem_final, b.mem_final)
    H.assert_close("grad_I", H.lanes_2d(a.grad_I), H.lanes_2d(b.grad_I), *H.TOL[w.io_dtype])


def test_rleaky_zero_reset_is_unsupported(cuda_device):
    w = W.RLEAKY_C6.scaled(T=2, B=2, N=8, reset="zero")
    layer = snn.ScanLayer(w, device=cuda_device)
    inp = {k: t.to(cuda_device) for k, t in W.make_scan_inputs(w).items()}
    with pytest.raises(snn.SnnError):
        layer.forward(inp["I"], inp["beta"], inp["thr"], v=inp["v"])


def test_rleaky_full_size(cuda_device):
    w = W.RLEAKY_C6
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    H.check_all(w, inp, layer, H.oracle_expect(w, inp))


@pytest.mark.parametrize("save,k", [("recompute", 16), ("mem", 8)])
def test_rleaky_full_size_large_bf16(save, k, cuda_device):
    w = W.RLEAKY_C7.scaled(save=save, ckpt_every=k)
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    check_every_lane_in_blocks(w, inp, layer)


# ---------------------------------------------------------------------------
# Recompute BPTT with the replayed segment in registers (8-, 12- and 16-step
# checkpoint segments of the Leaky and recurrent Leaky neurons)
# ---------------------------------------------------------------------------

SEG_CASES = [
    # T, B, N, K: a short first segment, one segment shorter than K, T = K,
    # several CTAs with a ragged last strip
    (37, 3, 1368, 16), (9, 4, 1000, 16), (16, 2, 2048, 16), (40, 5, 1000, 8),
    (5, 7, 1000, 8), (64, 16, 8192, 16), (33, 9, 4096, 8), (29, 3, 1368, 12),
    (12, 2, 2048, 12), (50, 6, 4096, 12),
]


# The per-neuron parameter-gradient reduction, bit for bit against its
# stated summation order: T, B, N, K, neuron.  One sample; B not a multiple
# of the 8 splits; 64 samples; a width below one warp's 32 neurons and a
# ragged last block; the recurrent neuron's v; the register-segment BPTT (K
# 8, 12, 16) and the shared-memory replay (K = 5), store mode in between.
REDUCE_CASES = [(24, 1, 2048, 8, "leaky"), (17, 3, 4096, 8, "leaky"), (40, 64, 1024, 12, "leaky"),
                (9, 5, 20, 8, "rleaky"), (33, 11, 8192, 16, "rleaky"), (20, 9, 1000, 5, "leaky"),
                (12, 10, 200, 0, "leaky")]


def two_add(hi, lo, x):
    """(hi, lo) += x in float32, the rounding error of hi + x kept in lo
    (Knuth's two-sum, every operation rounded to nearest)."""
    f = np.float32
    s = (hi + x).astype(f)
    z = (s - hi).astype(f)
    e = ((hi - (s - z).astype(f)).astype(f) + (x - z).astype(f)).astype(f)
    return s, (lo + e).astype(f)


def neuron_order_sum(part, B, N):
    """The order the per-neuron sum takes on the GPU: split s of the samples,
    [B*s/S, B*(s+1)/S) with S = min(B, 8), added in fp32 in sample order; the
    S split sums added in split order, compensated (two-sum); the sum plus
    its error rounded to fp32 (a non-finite sum as it is)."""
    S = min(B, 8)
    hi = np.zeros(N, np.float32)
    lo = np.zeros(N, np.float32)
    for s in range(S):
        acc = np.zeros(N, np.float32)
        for b in range(B * s // S, B * (s + 1) // S):
            acc = (acc + part[b]).astype(np.float32)
        hi, lo = two_add(hi, lo, acc)
    with np.errstate(invalid="ignore"):
        return np.where(np.isfinite(hi), (hi + lo).astype(np.float32), hi)


@pytest.mark.parametrize("case", range(len(REDUCE_CASES)))
def test_per_neuron_reduction_order(case, cuda_device):
    T, B, N, K, neuron = REDUCE_CASES[case]
    dt = W.BF16 if K in (12, 16) else [W.BF16, W.F32][case % 2]
    w = W.ScanWorkload(
        name=f"reduce_{case}", neuron=neuron, T=T, B=B, N=N, C=4, HW=max(1, N // 4), in_dtype=dt,
        io_dtype=dt, i_mean=0.5, i_std=0.6, beta=("uniform", 0.5, 0.95),
        thr=("uniform", 0.6, 1.4), v=("uniform", -0.6, 0.6), beta_mode="per_neuron",
        thr_mode="per_neuron", v_mode="per_neuron", reset="subtract", detach_reset=True,
        surrogate="atan", sg_param=2.0, save="recompute" if K else "mem", ckpt_every=K or 8,
        want_mem=True, seed_index=700 + case)
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    H.check_all(w, inp, layer, H.oracle_expect(w, inp))
    # the reduction's order applied to the kernel's own per-lane partials
    # (workspace: a 256-byte status block, then one 256-byte-aligned partial
    # array per parameter)
    pnames = ["beta", "thr"] + (["v"] if neuron == "rleaky" else [])
    L = B * N
    lb = (L * 4 + 255) // 256 * 256
    ws = layer.ws.cpu().numpy()
    got = {}
    for k, pname in enumerate(pnames):
        part = ws[256 + k * lb: 256 + k * lb + 4 * L].view(np.float32).reshape(B, N)
        got[pname] = getattr(layer, f"grad_{pname}").cpu().numpy().copy()
        assert np.array_equal(got[pname], neuron_order_sum(part, B, N), equal_nan=True), pname
    # a second backward into cleared outputs writes the same bits
    for pname in pnames:
        getattr(layer, f"grad_{pname}").fill_(-1.0)
    d = {k: v.to("cuda") for k, v in inp.items()}
    layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], alpha=d.get("alpha"),
                   mem0=d.get("mem0"), grad_mem=d.get("grad_mem"),
                   grad_mem_final=d.get("grad_mem_final"), v=d.get("v"))
    torch.cuda.synchronize()
    assert layer.status() == 0
    for pname in pnames:
        assert np.array_equal(getattr(layer, f"grad_{pname}").cpu().numpy(), got[pname],
                              equal_nan=True), pname


# Scalar and per-channel parameter gradients through their reduction
# launches: T, B, N, C, HW, save, neuron.  Channel runs of one lane
# (channel-last) and of many; a synaptic neuron (alpha); the shared-memory
# recompute kernel; a shape small enough for the plain kernels.
PARAM_CASES = [(25, 8, 6912, 12, 576, "mem", "leaky"), (25, 16, 4096, 64, 1, "mem", "leaky"),
               (30, 4, 4096, 16, 256, "mem", "synaptic"), (33, 5, 1024, 8, 128, "recompute", "leaky"),
               (3, 2, 8, 2, 4, "mem", "leaky")]


@pytest.mark.parametrize("case", range(len(PARAM_CASES)))
def test_scalar_and_channel_gradients(case, cuda_device):
    """The oracle's parameter gradients, and the same bits from a second
    backward into cleared outputs (every completion ticket back at zero)."""
    T, B, N, C, HW, save, neuron = PARAM_CASES[case]
    dt = [W.F32, W.BF16][case % 2]
    w = W.ScanWorkload(
        name=f"pfold_{case}", neuron=neuron, T=T, B=B, N=N, C=C, HW=HW, in_dtype=dt,
        io_dtype=dt, i_mean=0.5, i_std=0.6, beta=("uniform", 0.5, 0.95),
        thr=("uniform", 0.6, 1.4), alpha=("uniform", 0.5, 0.9),
        beta_mode=["per_channel", "scalar"][case % 2], thr_mode=["scalar", "per_channel"][case % 2],
        alpha_mode="per_channel", reset=["zero", "subtract"][case % 2], detach_reset=True,
        surrogate="fast_sigmoid", sg_param=25.0, save=save, ckpt_every=3, want_mem=True,
        seed_index=800 + case)
    inp = W.make_scan_inputs(w)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    H.check_all(w, inp, layer, H.oracle_expect(w, inp))
    pnames = ["beta", "thr"] + (["alpha"] if neuron == "synaptic" else [])
    got = {p: getattr(layer, f"grad_{p}").clone() for p in pnames}
    for p in pnames:
        getattr(layer, f"grad_{p}").fill_(-1.0)
    d = {k: v.to("cuda") for k, v in inp.items()}
    layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], alpha=d.get("alpha"),
                   mem0=d.get("mem0"), syn0=d.get("syn0"), grad_mem=d.get("grad_mem"),
                   grad_mem_final=d.get("grad_mem_final"),
                   grad_syn_final=d.get("grad_syn_final"))
    torch.cuda.synchronize()
    assert layer.status() == 0
    for p in pnames:
        assert torch.equal(getattr(layer, f"grad_{p}"), got[p]), p


@pytest.mark.parametrize("neuron", ["leaky", "rleaky"])
@pytest.mark.parametrize("case", range(len(SEG_CASES)))
def test_register_segment_recompute(case, neuron, cuda_device):
    T, B, N, K = SEG_CASES[case]
    dt = [W.BF16, W.F16, W.F32][case % 3] if K == 8 else [W.BF16, W.F16][case % 2]
    reset = "subtract" if neuron == "rleaky" else ["subtract", "zero"][case % 2]
    w = W.ScanWorkload(
        name=f"seg_{neuron}_{case}", neuron=neuron, T=T, B=B, N=N, C=8, HW=N // 8,
        in_dtype=dt, io_dtype=dt, i_mean=0.5, i_std=0.6, beta=("uniform", 0.5, 0.95),
        thr=("uniform", 0.6, 1.4), v=("uniform", -0.6, 0.6), beta_mode=MODES[case % 3],
        thr_mode=MODES[(case + 1) % 3], v_mode=MODES[(case + 2) % 3], reset=reset,
        detach_reset=(case % 2 == 0), surrogate=["fast_sigmoid", "atan"][case % 2],
        sg_param=[25.0, 2.0][case % 2], save="recompute", ckpt_every=K, want_mem=True,
        seed_index=500 + case)
    opts = dict(with_mem0=(case % 2 == 1), with_grad_mem=(case % 3 == 2),
                with_grad_final=(case % 2 == 0))
    inp = W.make_scan_inputs(w, **opts)
    layer = H.run_gpu(w, inp)
    assert layer.status() == 0
    H.check_all(w, inp, layer, H.oracle_expect(w, inp))
    # the shared-memory replay kernel on the same inputs: same spike path, the
    # reverse passes agree within the fp32 gradient tolerance
    old = H.run_gpu(w, inp, debug_flags=snn.DEBUG_NO_SEGMENT)
    assert old.status() == 0
    assert torch.equal(layer.spk, old.spk)
    if layer.ckpt is not None:  # T > K: checkpoints exist
        assert torch.equal(layer.ckpt, old.ckpt)
    H.assert_close("grad_I", H.lanes_2d(layer.grad_I), H.lanes_2d(old.grad_I), *H.TOL[w.io_dtype])
