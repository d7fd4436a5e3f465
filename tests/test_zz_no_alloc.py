"""The Leaky BPTT entry point that allocates nothing, through the C ABI.

snn_leaky_bwd_noalloc serves callers that cannot allocate device memory (a
host whose device memory another runtime budgets, a real-time loop that must
not call cudaMalloc, a C host without an allocator): its workspace is a fixed
array inside the library.  It must give exactly the results of snn_leaky_bwd
on a freshly initialised workspace -- the same kernels in the same order, so
bit for bit -- whatever the previous call on the shared array was: the same
shape, another shape or parameter layout (the reductions' tickets then sit
at other offsets), or a call whose wait gave up.  Kept in a file of its own
that pytest collects last.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2211_10725_gb300 import build_lib, snn
from paper_2211_10725_gb300 import workloads as W
from tests import scan_harness as H

pytestmark = pytest.mark.gpu

SNN_ERR_WORKSPACE = 4
SNN_ERR_TIMEOUT = 6
OUTS = ("grad_I", "grad_beta", "grad_thr", "grad_mem0")


class Case:
    """A Leaky workload run forward and backward through the workspace entry
    point (the reference results), ready for no-allocation backward calls."""

    def __init__(self, w, device, **desc_over):
        self.w = w
        self.inp = W.make_scan_inputs(w, with_mem0=True, with_grad_final=True)
        self.d = {k: v.to(device) for k, v in self.inp.items()}
        self.layer = snn.ScanLayer(w, device=device, **desc_over)
        d = self.d
        self.layer.forward(d["I"], d["beta"], d["thr"], mem0=d["mem0"])
        self.layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], mem0=d["mem0"],
                            grad_mem_final=d["grad_mem_final"])
        torch.cuda.synchronize()
        assert self.layer.status() == 0
        self.ref = {k: getattr(self.layer, k).clone() for k in OUTS}
        self.device = device

    def noalloc(self, desc=None):
        """One snn_leaky_bwd_noalloc call into fresh (NaN-filled) outputs;
        returns (outputs, kernel status)."""
        L, d = self.layer, self.d
        out = {k: torch.full_like(self.ref[k], float("nan")) for k in OUTS}
        status = torch.full((1,), -1, dtype=torch.int32, device=self.device)
        recompute = self.w.save == "recompute"
        snn.snn_leaky_bwd_noalloc(desc or L.desc, d["I"] if recompute else None, L.ckpt, L.mem,
                                  L.spk, d["beta"], d["thr"], d["mem0"], d["grad_spk"], None,
                                  d["grad_mem_final"], out["grad_I"], out["grad_beta"],
                                  out["grad_thr"], out["grad_mem0"], status=status)
        torch.cuda.synchronize()
        return out, int(status.item())

    def check(self, out):
        """Bit for bit against the workspace entry point, and within the
        scan tolerances against the oracle."""
        for k in OUTS:
            assert torch.equal(out[k], self.ref[k]), f"{k} differs from snn_leaky_bwd"
        w, ref = self.w, H.oracle_expect(self.w, self.inp)
        rtol, atol = H.TOL[w.io_dtype]
        H.assert_close("grad_I", H.lanes_2d(out["grad_I"]), ref["grad_I"], rtol, atol,
                       ref["grad_I_scale"])
        f_rtol, f_atol = H.TOL[W.F32]
        H.assert_close("grad_mem0", H.lanes_1d(out["grad_mem0"]), ref["grad_mem0"], f_rtol,
                       f_atol, ref["grad_mem0_scale"])
        H.check_param_grad("grad_beta", H.lanes_1d(out["grad_beta"]), ref["grad_beta"],
                           ref["grad_beta_lane"], w.B, w.N, w.beta_mode, w.C, w.HW)
        H.check_param_grad("grad_thr", H.lanes_1d(out["grad_thr"]), ref["grad_thr"],
                           ref["grad_thr_lane"], w.B, w.N, w.thr_mode, w.C, w.HW)


@pytest.mark.parametrize("save", ["recompute", "mem"])
def test_noalloc_matches_workspace_entry_point(save, cuda_device):
    build_lib.build()
    case = Case(W.BIG_C5.scaled(T=64, B=16, save=save), cuda_device)
    for _ in range(2):  # two calls in a row: the shared array keeps the last call's contents
        out, status = case.noalloc()
        assert status == 0
        case.check(out)


def test_noalloc_after_shape_and_layout_changes(cuda_device):
    """A large per-neuron call, then a smaller one with scalar beta and
    per-channel thr (its tickets land where the first call left partials),
    then the first again: each exact against a fresh workspace."""
    a = Case(W.BIG_C5.scaled(T=40, B=16, save="recompute"), cuda_device)
    b = Case(W.BIG_C5.scaled(name="noalloc_small", T=24, B=8, N=2048, C=16, HW=128,
                             beta=("const", 0.9), beta_mode="scalar", thr_mode="per_channel",
                             save="mem"), cuda_device)
    c = Case(W.BIG_C5.scaled(name="noalloc_chlast", T=12, B=4, N=1536, C=8, HW=1,
                             beta_mode="per_channel", thr_mode="per_channel", reset="zero",
                             save="recompute", ckpt_every=4), cuda_device)
    for case in (a, b, c, a, c, b):
        out, status = case.noalloc()
        assert status == 0
        case.check(out)


def test_noalloc_after_a_timeout(cuda_device):
    """A call whose producer issues nothing gives up its waits (status
    SNN_ERR_TIMEOUT, no fault); the next normal call on the same array is
    exact."""
    case = Case(W.BIG_C5.scaled(T=32, B=8, save="recompute"), cuda_device)
    idle = snn.make_desc(case.w, debug_flags=snn.DEBUG_PRODUCER_IDLE, wait_limit_ns=2_000_000)
    _, status = case.noalloc(idle)
    assert status == SNN_ERR_TIMEOUT
    out, status = case.noalloc()
    assert status == 0
    case.check(out)


def test_noalloc_rejects_workspace_beyond_its_scratch(cuda_device):
    lib = snn.load_library()
    d = snn.make_desc(W.BIG_C5.scaled(B=256))  # 2M lanes: workspace > 16 MiB
    assert snn.snn_scan_workspace_bytes(d) > (16 << 20)
    args = [16] * 14 + [None, None]
    assert lib.snn_leaky_bwd_noalloc(ctypes.byref(d), *args) == SNN_ERR_WORKSPACE
