"""Host-side checks of the C ABI (no GPU needed): the library loads, exports
every function include/snn.h declares, and rejects bad arguments before it
touches CUDA."""
import ctypes

import pytest

from paper_2211_10725_gb300 import build_lib, snn
from paper_2211_10725_gb300 import workloads as W


@pytest.fixture(scope="module")
def lib():
    build_lib.build()
    return snn.load_library()


def test_exports_every_declared_function(lib):
    names = snn.header_functions()
    assert len(names) >= 11
    for n in names:
        assert hasattr(lib, n), n
    # and the binding declares a signature for each
    assert set(names) <= set(snn._SIGS)


def test_descriptor_layout_matches(lib):
    assert lib.snn_scan_desc_size() == ctypes.sizeof(snn.ScanDesc)


def test_status_strings(lib):
    for code, name in snn.STATUS_NAMES.items():
        assert snn.status_string(code).startswith(name)
    assert snn.status_string(99).startswith("SNN_ERR_UNKNOWN")


def test_workspace_and_ckpt_sizes(lib):
    d = snn.make_desc(W.BIG_C5)
    L = W.BIG_C5.B * W.BIG_C5.N
    ws = snn.snn_scan_workspace_bytes(d)
    assert ws >= 3 * 4 * L
    assert snn.snn_scan_ckpt_elems(d, False) == (500 // 8) * L      # ceil(500/8)-1 = 62
    assert snn.snn_scan_ckpt_elems(d, True) == 2 * (500 // 8) * L
    d2 = snn.make_desc(W.LEAKY_C1)
    assert snn.snn_scan_ckpt_elems(d2, False) == 0                 # store variant


@pytest.mark.parametrize("field,value", [
    ("T", -1), ("B", -2), ("in_dtype", 7), ("reset", 3), ("detach_reset", 2),
    ("surrogate", 5), ("beta_mode", 9), ("save", 4), ("reserved0", 1),
    ("wait_limit_ns", -5)])
def test_invalid_descriptor_rejected(lib, field, value):
    d = snn.make_desc(W.LEAKY_C1, **{field: value})
    assert snn.snn_scan_workspace_bytes(d) == 0
    st = lib.snn_leaky_fwd(ctypes.byref(d), 16, 16, 16, None, 16, 16, None, None, 16, 1 << 30, None)
    assert st == 1


def test_bad_sg_param_and_per_channel_shape(lib):
    d = snn.make_desc(W.LEAKY_C1, sg_param=0.0)
    assert snn.snn_scan_workspace_bytes(d) == 0
    d = snn.make_desc(W.CONV_C4A, HW=7)          # N is not a multiple of C*HW
    assert snn.snn_scan_workspace_bytes(d) == 0
    d = snn.make_desc(W.BIG_C5, ckpt_every=0)
    assert snn.snn_scan_workspace_bytes(d) == 0


def test_unsupported_combinations(lib):
    d = snn.make_desc(W.LEAKY_C1, in_dtype=1, io_dtype=0)       # bf16 in, fp32 out
    st = lib.snn_leaky_fwd(ctypes.byref(d), 16, 16, 16, None, 16, 16, None, None, 16, 1 << 30, None)
    assert st == 3
    d = snn.make_desc(W.BIG_C5, ckpt_every=65)
    assert snn.snn_scan_workspace_bytes(d) == 0


def test_null_and_misaligned_pointers(lib):
    d = snn.make_desc(W.LEAKY_C1)
    big = 1 << 30
    f = lib.snn_leaky_fwd
    # missing I / spk / mem (store variant) / beta
    assert f(ctypes.byref(d), None, 16, 16, None, 16, 16, None, None, 16, big, None) == 1
    assert f(ctypes.byref(d), 16, 16, 16, None, None, 16, None, None, 16, big, None) == 1
    assert f(ctypes.byref(d), 16, 16, 16, None, 16, None, None, None, 16, big, None) == 1
    assert f(ctypes.byref(d), 16, None, 16, None, 16, 16, None, None, 16, big, None) == 1
    # misaligned device pointers
    assert f(ctypes.byref(d), 24, 16, 16, None, 16, 16, None, None, 16, big, None) == 2
    assert f(ctypes.byref(d), 16, 16, 16, 20, 16, 16, None, None, 16, big, None) == 2
    # workspace missing or too small
    assert f(ctypes.byref(d), 16, 16, 16, None, 16, 16, None, None, None, big, None) == 4
    assert f(ctypes.byref(d), 16, 16, 16, None, 16, 16, None, None, 16, 64, None) == 4
    # the recompute variant needs its checkpoint buffer
    d5 = snn.make_desc(W.BIG_C5)
    assert f(ctypes.byref(d5), 16, 16, 16, None, 16, None, None, None, 16, big, None) == 1


BWD_ARGS = ["I", "ckpt", "mem", "spk", "beta", "thr", "mem0", "grad_spk", "grad_mem",
            "grad_mem_final", "grad_I", "grad_beta", "grad_thr", "grad_mem0", "ws"]


def _bwd(lib, d, **ptrs):
    vals = [ptrs.get(k) for k in BWD_ARGS]
    return lib.snn_leaky_bwd(ctypes.byref(d), *vals, 1 << 30, None)


def test_backward_argument_checks(lib):
    good = dict(mem=16, spk=16, beta=16, thr=16, grad_spk=16, grad_I=16, ws=16)
    d = snn.make_desc(W.LEAKY_C1)
    for missing in ("mem", "beta", "thr", "grad_spk", "grad_I"):
        p = dict(good)
        p.pop(missing)
        assert _bwd(lib, d, **p) == 1, missing
    p = dict(good)
    p["grad_beta"] = 8
    assert _bwd(lib, d, **p) == 2
    # fp32 store variant may omit spk; a half-precision one may not
    p = dict(good)
    p.pop("spk")
    assert _bwd(lib, snn.make_desc(W.LEAKY_C1, in_dtype=1, io_dtype=1), **p) == 1
    # recompute variant needs I and the checkpoints
    d5 = snn.make_desc(W.BIG_C5)
    rec = dict(beta=16, thr=16, grad_spk=16, grad_I=16, ws=16, I=16)
    assert _bwd(lib, d5, **rec) == 1
    rec = dict(beta=16, thr=16, grad_spk=16, grad_I=16, ws=16, ckpt=16)
    assert _bwd(lib, d5, **rec) == 1


# The fused entry points check their arguments before any CUDA call.  The
# pointers below are never dereferenced: every call here is rejected first.
def _fused_desc(**over):
    w = W.ScanWorkload(name="fused", neuron="leaky", T=25, B=16, N=64, in_dtype=W.F32,
                       io_dtype=W.BF16, save="mem", want_mem=True)
    return snn.make_desc(w, **over)


def test_dense_leaky_fwd_argument_checks(lib):
    f = lambda d, P=1, K=64, X=16, ws_bytes=256: lib.snn_dense_leaky_fwd(
        ctypes.byref(d), P, K, X, 16, 16, 16, 16, 16, None, 16, ws_bytes, None)
    assert f(_fused_desc(T=129)) == 3                  # a tile holds every step
    assert f(_fused_desc(io_dtype=0)) == 3             # bf16 storage only
    assert f(_fused_desc(save=1, ckpt_every=8)) == 3   # the trace is stored
    assert f(_fused_desc(), K=12) == 3                 # 16-byte rows
    assert f(_fused_desc(N=12)) == 3
    assert f(_fused_desc(), P=3) == 1                  # N % P
    assert f(_fused_desc(reset=3)) == 1
    assert f(_fused_desc(), X=None) == 1
    assert f(_fused_desc(), X=24) == 2
    assert f(_fused_desc(), ws_bytes=64) == 4


def test_dense_leaky_bwd_argument_checks(lib):
    def f(d, K=64, dI=16, Wp=16, spk=16, ckpt=None, ws_bytes=256):
        return lib.snn_dense_leaky_bwd(ctypes.byref(d), K, dI, Wp, 16, 16, 16, spk, ckpt, 16,
                                       16, ws_bytes, None)
    assert f(_fused_desc(T=129)) == 3
    assert f(_fused_desc(io_dtype=0)) == 3
    assert f(_fused_desc(save=1, ckpt_every=8)) == 3
    assert f(_fused_desc(), K=12) == 3
    assert f(_fused_desc(N=12)) == 3
    assert f(_fused_desc(beta_mode=2, C=64, HW=1)) == 3   # scalar or per neuron only
    assert f(_fused_desc(surrogate=5)) == 1
    assert f(_fused_desc(sg_param=0.0)) == 1
    assert f(_fused_desc(), spk=None, ckpt=None) == 1     # no spike source
    assert f(_fused_desc(), Wp=None) == 1
    assert f(_fused_desc(), dI=24) == 2
    assert f(_fused_desc(), ckpt=40) == 2
    assert f(_fused_desc(), ws_bytes=64) == 4


def test_rate_ce_leaky_bwd_argument_checks(lib):
    need = snn.snn_rate_ce_workspace_bytes(16)

    def f(d, C=10, pop=1, total=0, spk=16, mem=16, ws_bytes=need):
        return lib.snn_rate_ce_leaky_bwd(ctypes.byref(d), C, pop, total, spk, 16, 16, 16, mem,
                                         None, 16, None, 16, 16, ws_bytes, None)
    assert f(_fused_desc(), C=10, pop=7) == 1             # C * pop > ld
    assert f(_fused_desc(), total=8) == 1                 # batch_total < B
    assert f(_fused_desc(), C=2000) == 1                  # at most 1024 classes
    assert f(_fused_desc(save=1, ckpt_every=8)) == 3      # needs the stored trace
    assert f(_fused_desc(thr_mode=2, C=64, HW=1)) == 3
    assert f(_fused_desc(io_dtype=7)) == 1
    assert f(_fused_desc(reset=3)) == 1
    assert f(_fused_desc(), mem=None) == 1
    assert f(_fused_desc(), spk=24) == 2
    assert f(_fused_desc(), ws_bytes=64) == 4
