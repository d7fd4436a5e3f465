"""The no-allocation Leaky BPTT entry point (for callers that cannot
allocate device memory) against the workspace entry point, through the C
ABI.  Kept in a file of its own that pytest collects last."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2211_10725_gb300 import build_lib, snn
from paper_2211_10725_gb300 import workloads as W
from tests import scan_harness as H

pytestmark = pytest.mark.gpu


def _outputs(layer, device):
    w = layer.w
    nan = float("nan")
    return {
        "grad_I": torch.full_like(layer.grad_I, nan),
        "grad_beta": torch.full_like(layer.grad_beta, nan),
        "grad_thr": torch.full_like(layer.grad_thr, nan),
        "grad_mem0": torch.full((w.B, w.N), nan, dtype=torch.float32, device=device),
    }


@pytest.mark.parametrize("save", ["recompute", "mem"])
def test_noalloc_matches_workspace_entry_point(save, cuda_device):
    build_lib.build()
    lib = snn.load_library()
    w = W.BIG_C5.scaled(T=64, B=16, save=save)
    inp = W.make_scan_inputs(w, with_mem0=True, with_grad_final=True)
    d = {k: v.to(cuda_device) for k, v in inp.items()}
    layer = snn.ScanLayer(w, device=cuda_device)
    layer.forward(d["I"], d["beta"], d["thr"], mem0=d["mem0"])
    layer.backward(d["I"], d["beta"], d["thr"], d["grad_spk"], mem0=d["mem0"],
                   grad_mem_final=d["grad_mem_final"])
    torch.cuda.synchronize()
    assert layer.status() == 0
    ref = {k: getattr(layer, k).clone() for k in ("grad_I", "grad_beta", "grad_thr", "grad_mem0")}
    recompute = save == "recompute"
    rtol, atol = H.TOL[w.io_dtype]
    for _ in range(2):  # two calls in a row: the shared scratch keeps the last call's contents
        out = _outputs(layer, cuda_device)
        status = torch.full((1,), -1, dtype=torch.int32, device=cuda_device)
        snn.snn_leaky_bwd_noalloc(layer.desc, d["I"] if recompute else None, layer.ckpt,
                                  layer.mem, layer.spk, d["beta"], d["thr"], d["mem0"],
                                  d["grad_spk"], None, d["grad_mem_final"], out["grad_I"],
                                  out["grad_beta"], out["grad_thr"], out["grad_mem0"],
                                  status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        H.assert_close("grad_I", H.lanes_2d(out["grad_I"]), H.lanes_2d(ref["grad_I"]), rtol, atol)
        for k in ("grad_beta", "grad_thr", "grad_mem0"):
            H.assert_close(k, H.lanes_1d(out[k]), H.lanes_1d(ref[k]), *H.TOL[W.F32])


def test_noalloc_rejects_workspace_beyond_its_scratch(cuda_device):
    lib = snn.load_library()
    d = snn.make_desc(W.BIG_C5.scaled(B=256))  # 2M lanes: workspace > 16 MiB
    assert snn.snn_scan_workspace_bytes(d) > (16 << 20)
    args = [16] * 14 + [None, None]
    assert lib.snn_leaky_bwd_noalloc(ctypes.byref(d), *args) == 4   # SNN_ERR_WORKSPACE
