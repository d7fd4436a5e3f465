"""ctypes binding of libsnn (include/snn.h).

The functions named like the C entry points marshal torch tensors into
device pointers and call the library; every step of the scan runs in the
library's CUDA kernels.  PyTorch only allocates memory and supplies the
current stream.  If the library is missing the binding raises: there is no
fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional

import torch

from . import workloads as W

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_lib", "libsnn.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "snn.h")

SNN_OK = 0
STATUS_NAMES = {0: "SNN_OK", 1: "SNN_ERR_INVALID_ARG", 2: "SNN_ERR_ALIGNMENT",
                3: "SNN_ERR_UNSUPPORTED", 4: "SNN_ERR_WORKSPACE", 5: "SNN_ERR_CUDA",
                6: "SNN_ERR_TIMEOUT"}
DTYPE_CODE = {W.F32: 0, W.BF16: 1, W.F16: 2}
RESET_CODE = {"subtract": 0, "zero": 1, "none": 2}
SG_CODE = {"fast_sigmoid": 0, "atan": 1}
PMODE_CODE = {"scalar": 0, "per_neuron": 1, "per_channel": 2}
SAVE_CODE = {"mem": 0, "recompute": 1}
DEBUG_PRODUCER_IDLE = 1
DEBUG_FORCE_PLAIN = 2
DEBUG_NO_SEGMENT = 4


class SnnError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}")


class ScanDesc(ctypes.Structure):
    """Mirror of snn_scan_desc."""
    _fields_ = [
        ("T", ctypes.c_int64), ("B", ctypes.c_int64), ("N", ctypes.c_int64),
        ("C", ctypes.c_int64), ("HW", ctypes.c_int64),
        ("in_dtype", ctypes.c_int32), ("io_dtype", ctypes.c_int32),
        ("reset", ctypes.c_int32), ("detach_reset", ctypes.c_int32),
        ("surrogate", ctypes.c_int32), ("sg_param", ctypes.c_float),
        ("beta_mode", ctypes.c_int32), ("thr_mode", ctypes.c_int32),
        ("alpha_mode", ctypes.c_int32), ("save", ctypes.c_int32),
        ("ckpt_every", ctypes.c_int32), ("reserved0", ctypes.c_int32),
        ("wait_limit_ns", ctypes.c_int64), ("debug_flags", ctypes.c_uint32),
        ("reserved1", ctypes.c_uint32),
    ]


_P = ctypes.c_void_p
_SIGS = {
    "snn_status_string": ([ctypes.c_int], ctypes.c_char_p),
    "snn_version": ([], ctypes.c_int),
    "snn_scan_desc_size": ([], ctypes.c_size_t),
    "snn_scan_workspace_bytes": ([ctypes.POINTER(ScanDesc)], ctypes.c_size_t),
    "snn_scan_ckpt_elems": ([ctypes.POINTER(ScanDesc), ctypes.c_int], ctypes.c_int64),
    "snn_workspace_init": ([_P, ctypes.c_size_t, _P], ctypes.c_int),
    "snn_workspace_status": ([_P, _P], ctypes.c_int),
    "snn_leaky_fwd": ([ctypes.POINTER(ScanDesc)] + [_P] * 9 + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_leaky_bwd": ([ctypes.POINTER(ScanDesc)] + [_P] * 15 + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_synaptic_fwd": ([ctypes.POINTER(ScanDesc)] + [_P] * 13 + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_synaptic_bwd": ([ctypes.POINTER(ScanDesc)] + [_P] * 21 + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_leaky_bwd_noalloc": ([ctypes.POINTER(ScanDesc)] + [_P] * 16, ctypes.c_int),
    "snn_rleaky_fwd": ([ctypes.POINTER(ScanDesc)] + [_P] * 10 + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_rleaky_bwd": ([ctypes.POINTER(ScanDesc)] + [_P] * 17 + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_dense_layer_fwd": ([ctypes.c_int64] * 3 + [_P] * 4 + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_dense_workspace_bytes": ([ctypes.c_int64] * 3, ctypes.c_size_t),
    "snn_dense_layer_bwd": ([ctypes.c_int64] * 3 + [_P] * 6 + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_rate_ce_workspace_bytes": ([ctypes.c_int64], ctypes.c_size_t),
    "snn_kernel_launches": ([], ctypes.c_uint64),
    "snn_dense_leaky_bwd": ([ctypes.POINTER(ScanDesc), ctypes.c_int64] + [_P] * 9
                            + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_dense_leaky_fwd": ([ctypes.POINTER(ScanDesc), ctypes.c_int64, ctypes.c_int64] + [_P] * 8
                            + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_conv2d_small_fwd_nhwc": ([ctypes.c_int64] * 8 + [_P] * 4, ctypes.c_int),
    "snn_conv2d_small_dw_workspace_bytes": ([ctypes.c_int64] * 7, ctypes.c_size_t),
    "snn_conv2d_small_dw_nhwc": ([ctypes.c_int64] * 8 + [_P] * 4 + [ctypes.c_size_t, _P],
                                 ctypes.c_int),
    "snn_im2col_nhwc": ([ctypes.c_int64] * 7 + [_P] * 3, ctypes.c_int),
    "snn_col2im_nhwc": ([ctypes.c_int64] * 7 + [_P] * 3, ctypes.c_int),
    "snn_maxpool2_fwd_nhwc": ([ctypes.c_int64] * 4 + [_P] * 4, ctypes.c_int),
    "snn_maxpool2_bwd_nhwc": ([ctypes.c_int64] * 4 + [_P] * 4, ctypes.c_int),
    "snn_rate_ce_loss": ([ctypes.c_int64] * 6 + [ctypes.c_int32] + [_P] * 5 + [ctypes.c_size_t, _P],
                         ctypes.c_int),
    "snn_rate_ce_leaky_bwd": ([ctypes.POINTER(ScanDesc)] + [ctypes.c_int64] * 3 + [_P] * 10
                              + [ctypes.c_size_t, _P], ctypes.c_int),
    "snn_adamw_step": ([ctypes.c_int64] + [_P] * 5 + [ctypes.c_float] * 5 + [ctypes.c_int64] +
                       [_P, _P], ctypes.c_int),
}

_lib: Optional[ctypes.CDLL] = None


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libsnn.so (built by paper_2211_10725_gb300.build_lib); raise if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"libsnn.so not built ({path}); run __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    for name, (args, res) in _SIGS.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    _lib = lib
    return lib


def header_functions(path: str = HEADER) -> list:
    """Names of the functions include/snn.h declares."""
    txt = open(path).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(snn_[a-z0-9_]+)\s*\(", txt)))


def status_string(status: int) -> str:
    return load_library().snn_status_string(status).decode()


def _check(status: int, where: str):
    if status != SNN_OK:
        raise SnnError(status, where)


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_desc(w: W.ScanWorkload, **over) -> ScanDesc:
    """Descriptor for a workload (fields can be overridden by keyword)."""
    d = ScanDesc()
    d.T, d.B, d.N, d.C, d.HW = w.T, w.B, w.N, w.C, w.HW
    d.in_dtype, d.io_dtype = DTYPE_CODE[w.in_dtype], DTYPE_CODE[w.io_dtype]
    d.reset = RESET_CODE[w.reset]
    d.detach_reset = 1 if w.detach_reset else 0
    d.surrogate = SG_CODE[w.surrogate]
    d.sg_param = w.sg_param
    d.beta_mode, d.thr_mode = PMODE_CODE[w.beta_mode], PMODE_CODE[w.thr_mode]
    d.alpha_mode = PMODE_CODE[w.v_mode if w.neuron == "rleaky" else w.alpha_mode]
    d.save = SAVE_CODE[w.save]
    d.ckpt_every = w.ckpt_every if w.save == "recompute" else 0
    for k, v in over.items():
        setattr(d, k, v)
    return d


# ---------------------------------------------------------------------------
# Thin wrappers with the C names (tensor -> pointer marshalling only)
# ---------------------------------------------------------------------------

def snn_scan_workspace_bytes(desc: ScanDesc) -> int:
    return load_library().snn_scan_workspace_bytes(ctypes.byref(desc))


def snn_scan_ckpt_elems(desc: ScanDesc, synaptic: bool) -> int:
    return load_library().snn_scan_ckpt_elems(ctypes.byref(desc), 1 if synaptic else 0)


def snn_workspace_init(ws: torch.Tensor, stream=None):
    _check(load_library().snn_workspace_init(_ptr(ws), ws.numel() * ws.element_size(),
                                             _stream(stream)), "snn_workspace_init")


def snn_workspace_status(ws: torch.Tensor, stream=None) -> int:
    return load_library().snn_workspace_status(_ptr(ws), _stream(stream))


def snn_leaky_fwd(desc, I, beta, thr, mem0, spk, mem, ckpt, mem_final, ws, stream=None):
    _check(load_library().snn_leaky_fwd(
        ctypes.byref(desc), _ptr(I), _ptr(beta), _ptr(thr), _ptr(mem0), _ptr(spk), _ptr(mem),
        _ptr(ckpt), _ptr(mem_final), _ptr(ws), ws.numel() * ws.element_size(),
        _stream(stream)), "snn_leaky_fwd")


def snn_leaky_bwd(desc, I, ckpt, mem, spk, beta, thr, mem0, grad_spk, grad_mem,
                  grad_mem_final, grad_I, grad_beta, grad_thr, grad_mem0, ws, stream=None):
    _check(load_library().snn_leaky_bwd(
        ctypes.byref(desc), _ptr(I), _ptr(ckpt), _ptr(mem), _ptr(spk), _ptr(beta), _ptr(thr),
        _ptr(mem0), _ptr(grad_spk), _ptr(grad_mem), _ptr(grad_mem_final), _ptr(grad_I),
        _ptr(grad_beta), _ptr(grad_thr), _ptr(grad_mem0), _ptr(ws),
        ws.numel() * ws.element_size(), _stream(stream)), "snn_leaky_bwd")


def snn_synaptic_fwd(desc, I, alpha, beta, thr, mem0, syn0, spk, mem, syn, ckpt, mem_final,
                     syn_final, ws, stream=None):
    _check(load_library().snn_synaptic_fwd(
        ctypes.byref(desc), _ptr(I), _ptr(alpha), _ptr(beta), _ptr(thr), _ptr(mem0),
        _ptr(syn0), _ptr(spk), _ptr(mem), _ptr(syn), _ptr(ckpt), _ptr(mem_final),
        _ptr(syn_final), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)),
        "snn_synaptic_fwd")


def snn_synaptic_bwd(desc, I, ckpt, mem, spk, syn, alpha, beta, thr, mem0, syn0, grad_spk,
                     grad_mem, grad_mem_final, grad_syn_final, grad_I, grad_alpha, grad_beta,
                     grad_thr, grad_mem0, grad_syn0, ws, stream=None):
    _check(load_library().snn_synaptic_bwd(
        ctypes.byref(desc), _ptr(I), _ptr(ckpt), _ptr(mem), _ptr(spk), _ptr(syn), _ptr(alpha),
        _ptr(beta), _ptr(thr), _ptr(mem0), _ptr(syn0), _ptr(grad_spk), _ptr(grad_mem),
        _ptr(grad_mem_final), _ptr(grad_syn_final), _ptr(grad_I), _ptr(grad_alpha),
        _ptr(grad_beta), _ptr(grad_thr), _ptr(grad_mem0), _ptr(grad_syn0), _ptr(ws),
        ws.numel() * ws.element_size(), _stream(stream)), "snn_synaptic_bwd")


def snn_rleaky_fwd(desc, I, v, beta, thr, mem0, spk, mem, ckpt, mem_final, ws, stream=None):
    _check(load_library().snn_rleaky_fwd(
        ctypes.byref(desc), _ptr(I), _ptr(v), _ptr(beta), _ptr(thr), _ptr(mem0), _ptr(spk),
        _ptr(mem), _ptr(ckpt), _ptr(mem_final), _ptr(ws), ws.numel() * ws.element_size(),
        _stream(stream)), "snn_rleaky_fwd")


def snn_rleaky_bwd(desc, I, ckpt, mem, spk, v, beta, thr, mem0, grad_spk, grad_mem,
                   grad_mem_final, grad_I, grad_v, grad_beta, grad_thr, grad_mem0, ws,
                   stream=None):
    _check(load_library().snn_rleaky_bwd(
        ctypes.byref(desc), _ptr(I), _ptr(ckpt), _ptr(mem), _ptr(spk), _ptr(v), _ptr(beta),
        _ptr(thr), _ptr(mem0), _ptr(grad_spk), _ptr(grad_mem), _ptr(grad_mem_final),
        _ptr(grad_I), _ptr(grad_v), _ptr(grad_beta), _ptr(grad_thr), _ptr(grad_mem0), _ptr(ws),
        ws.numel() * ws.element_size(), _stream(stream)), "snn_rleaky_bwd")


def snn_leaky_bwd_noalloc(desc, I, ckpt, mem, spk, beta, thr, mem0, grad_spk, grad_mem,
                          grad_mem_final, grad_I, grad_beta, grad_thr, grad_mem0, status=None,
                          stream=None):
    """Leaky BPTT using the library's fixed device scratch instead of a
    workspace, for callers that cannot allocate device memory."""
    _check(load_library().snn_leaky_bwd_noalloc(
        ctypes.byref(desc), _ptr(I), _ptr(ckpt), _ptr(mem), _ptr(spk), _ptr(beta), _ptr(thr),
        _ptr(mem0), _ptr(grad_spk), _ptr(grad_mem), _ptr(grad_mem_final), _ptr(grad_I),
        _ptr(grad_beta), _ptr(grad_thr), _ptr(grad_mem0), _ptr(status), _stream(stream)),
        "snn_leaky_bwd_noalloc")


def snn_dense_workspace_bytes(M: int, K: int, N: int) -> int:
    return load_library().snn_dense_workspace_bytes(M, K, N)


def snn_dense_layer_fwd(X, W, I, ws, stream=None):
    """I[M, N] = X[M, K] @ W[N, K]^T on the tensor cores (bf16 in, fp32 out)."""
    M, K = X.shape[-2], X.shape[-1]
    N = W.shape[0]
    _check(load_library().snn_dense_layer_fwd(M, K, N, _ptr(X), _ptr(W), _ptr(I), _ptr(ws),
                                              ws.numel() * ws.element_size(), _stream(stream)),
           "snn_dense_layer_fwd")


def snn_dense_layer_bwd(X, W, dI, dX, dW, ws, stream=None):
    """dX = dI @ W (bf16) and dW = dI^T @ X (fp32); either output may be None."""
    M, K = X.shape[-2], X.shape[-1]
    N = W.shape[0]
    _check(load_library().snn_dense_layer_bwd(M, K, N, _ptr(X), _ptr(W), _ptr(dI), _ptr(dX),
                                              _ptr(dW), _ptr(ws), ws.numel() * ws.element_size(),
                                              _stream(stream)), "snn_dense_layer_bwd")


class SideStream:
    """A second stream for launches off a training step's critical path (the
    weight-gradient products, which nothing waits on until the optimiser):
    fork() queues a call on it behind the work already queued on the main
    stream, join() makes the main stream wait for every call forked since the
    last join.  Both are event records and waits, so a captured CUDA graph
    holds them as fork and join edges."""

    def __init__(self, device=None):
        self.stream = torch.cuda.Stream(device)
        self._done = []

    def fork(self, main, call):
        """call(stream) on the side stream, after main's queued work."""
        main = torch.cuda.current_stream() if main is None else main
        ready = torch.cuda.Event()
        ready.record(main)
        self.stream.wait_event(ready)
        call(self.stream)
        done = torch.cuda.Event()
        done.record(self.stream)
        self._done.append(done)

    def join(self, main):
        main = torch.cuda.current_stream() if main is None else main
        for done in self._done:
            main.wait_event(done)
        self._done = []


def dense_layer_bwd_split(X, W, dI, dX, dW, ws, stream=None, side: Optional[SideStream] = None):
    """snn_dense_layer_bwd with, given a side stream, the weight gradient
    forked onto it (issued first, so it runs beside the input gradient,
    which the rest of the reverse pass waits on)."""
    if side is None or dW is None:
        snn_dense_layer_bwd(X, W, dI, dX, dW, ws, stream)
        return
    side.fork(stream, lambda st: snn_dense_layer_bwd(X, W, dI, None, dW, ws, st))
    if dX is not None:
        snn_dense_layer_bwd(X, W, dI, dX, None, ws, stream)


def snn_rate_ce_workspace_bytes(B: int) -> int:
    return load_library().snn_rate_ce_workspace_bytes(B)


def snn_rate_ce_loss(spk, labels, C, loss, grad_spk, ws=None, stream=None, batch_total=None,
                     pop=1):
    """Cross-entropy on output spike counts; spk/grad_spk [T, B, ld], C
    classes of pop neurons each.  The mean is over batch_total samples
    (default B: this batch).  ws: a zeroed uint8 device tensor of
    snn_rate_ce_workspace_bytes(B) bytes (a fresh one when None)."""
    T, B, ld = spk.shape
    dt = {torch.float32: 0, torch.bfloat16: 1, torch.float16: 2}[spk.dtype]
    if ws is None:
        ws = torch.zeros(snn_rate_ce_workspace_bytes(B), dtype=torch.uint8, device=spk.device)
    _check(load_library().snn_rate_ce_loss(T, B, C, pop, ld, batch_total or 0, dt, _ptr(spk),
                                           _ptr(labels), _ptr(loss), _ptr(grad_spk), _ptr(ws),
                                           ws.numel() * ws.element_size(), _stream(stream)),
           "snn_rate_ce_loss")


def snn_rate_ce_leaky_bwd(desc, spk, labels, C, beta, thr, mem, ckpt, loss, grad_spk, grad_I,
                          ws, stream=None, batch_total=None, pop=1):
    """snn_rate_ce_loss with the readout layer's BPTT in the same launch:
    writes loss, grad_I [T, B, ld] and (unless None) grad_spk.  ckpt: the
    forward's spike bits, or None to take the spike decisions from spk."""
    _check(load_library().snn_rate_ce_leaky_bwd(ctypes.byref(desc), C, pop, batch_total or 0,
                                                _ptr(spk), _ptr(labels), _ptr(beta), _ptr(thr),
                                                _ptr(mem), _ptr(ckpt), _ptr(loss), _ptr(grad_spk),
                                                _ptr(grad_I), _ptr(ws),
                                                ws.numel() * ws.element_size(), _stream(stream)),
           "snn_rate_ce_leaky_bwd")


def snn_adamw_step(w, w_bf16, grad, m, v, lr, beta1=0.9, beta2=0.999, eps=1e-8,
                   weight_decay=1e-2, step=1, step_counter=None, stream=None):
    """AdamW update in place of fp32 w, m, v from grad (same numel); writes
    the bf16 copy of the new weights to w_bf16 unless it is None.  With a
    device int64 [2] step_counter the step number is read from (and advanced
    on) the device instead of taken from ``step``."""
    n = w.numel()
    for t in (grad, m, v) + ((w_bf16,) if w_bf16 is not None else ()):
        if t.numel() != n:
            raise ValueError("snn_adamw_step: tensors differ in size")
    _check(load_library().snn_adamw_step(n, _ptr(w), _ptr(w_bf16), _ptr(grad), _ptr(m), _ptr(v),
                                         lr, beta1, beta2, eps, weight_decay, step,
                                         _ptr(step_counter), _stream(stream)), "snn_adamw_step")


def snn_dense_leaky_fwd(desc, X, W, beta, thr, spk, mem, ckpt, ws, P=1, stream=None):
    """GEMM of X [T*B*P, K] with W [Nout, K] and the Leaky scan of its
    currents in one kernel; writes spk, mem (and the spike bits to ckpt)."""
    K = X.shape[-1]
    _check(load_library().snn_dense_leaky_fwd(ctypes.byref(desc), P, K, _ptr(X), _ptr(W),
                                              _ptr(beta), _ptr(thr), _ptr(spk), _ptr(mem),
                                              _ptr(ckpt), _ptr(ws), ws.numel() * ws.element_size(),
                                              _stream(stream)), "snn_dense_leaky_fwd")


def snn_dense_leaky_bwd(desc, dI_up, W, beta, thr, mem, spk, ckpt, grad_I, ws, stream=None):
    """dX = dI_up [T*B, K] @ W [K, N] on the tensor cores, and the Leaky BPTT
    of the layer below on it in the same kernel; writes that layer's grad_I."""
    K = dI_up.shape[-1]
    _check(load_library().snn_dense_leaky_bwd(ctypes.byref(desc), K, _ptr(dI_up), _ptr(W),
                                              _ptr(beta), _ptr(thr), _ptr(mem), _ptr(spk),
                                              _ptr(ckpt), _ptr(grad_I), _ptr(ws),
                                              ws.numel() * ws.element_size(), _stream(stream)),
           "snn_dense_leaky_bwd")


def snn_kernel_launches() -> int:
    """Kernels the library has launched (or captured) in this process."""
    return int(load_library().snn_kernel_launches())


def snn_conv2d_small_fwd_nhwc(X, Wt, I, KH, KW, stream=None):
    """I [M, Ho, Wo, Cout] fp32 = X [M, H, W, Cin] (*) filters Wt [Cout, ldw]
    on the CUDA cores (few input channels)."""
    M, H, W_, Cin = X.shape
    Cout, ldw = Wt.shape
    _check(load_library().snn_conv2d_small_fwd_nhwc(M, H, W_, Cin, Cout, KH, KW, ldw, _ptr(X),
                                                    _ptr(Wt), _ptr(I), _stream(stream)),
           "snn_conv2d_small_fwd_nhwc")


def snn_conv2d_small_dw_workspace_bytes(M, H, W_, Cin, Cout, KH, KW) -> int:
    return load_library().snn_conv2d_small_dw_workspace_bytes(M, H, W_, Cin, Cout, KH, KW)


def snn_conv2d_small_dw_nhwc(X, dI, dW, KH, KW, ws, stream=None):
    """dW [Cout, ldw] fp32 of snn_conv2d_small_fwd_nhwc from dI [M, Ho, Wo, Cout] bf16."""
    M, H, W_, Cin = X.shape
    Cout, ldw = dW.shape
    _check(load_library().snn_conv2d_small_dw_nhwc(M, H, W_, Cin, Cout, KH, KW, ldw, _ptr(X),
                                                   _ptr(dI), _ptr(dW), _ptr(ws),
                                                   ws.numel() * ws.element_size(),
                                                   _stream(stream)), "snn_conv2d_small_dw_nhwc")


def snn_im2col_nhwc(X, cols, KH, KW, stream=None):
    """Patch rows of channel-last X [M, H, W, Cin] into cols [M*Ho*Wo, Kpad]."""
    M, H, W_, Cin = X.shape
    _check(load_library().snn_im2col_nhwc(M, H, W_, Cin, KH, KW, cols.shape[-1], _ptr(X),
                                          _ptr(cols), _stream(stream)), "snn_im2col_nhwc")


def snn_col2im_nhwc(dcols, dX, KH, KW, stream=None):
    """Patch-row gradient dcols [M*Ho*Wo, Kpad] summed onto dX [M, H, W, Cin]."""
    M, H, W_, Cin = dX.shape
    _check(load_library().snn_col2im_nhwc(M, H, W_, Cin, KH, KW, dcols.shape[-1], _ptr(dcols),
                                          _ptr(dX), _stream(stream)), "snn_col2im_nhwc")


def snn_maxpool2_fwd_nhwc(X, Y, idx, stream=None):
    M, H, W_, C = X.shape
    _check(load_library().snn_maxpool2_fwd_nhwc(M, H, W_, C, _ptr(X), _ptr(Y), _ptr(idx),
                                                _stream(stream)), "snn_maxpool2_fwd_nhwc")


def snn_maxpool2_bwd_nhwc(dY, idx, dX, stream=None):
    M, H, W_, C = dX.shape
    _check(load_library().snn_maxpool2_bwd_nhwc(M, H, W_, C, _ptr(dY), _ptr(idx), _ptr(dX),
                                                _stream(stream)), "snn_maxpool2_bwd_nhwc")


# ---------------------------------------------------------------------------
# A layer object: allocates the buffers of one scan workload on the device
# ---------------------------------------------------------------------------

class ScanLayer:
    """Device buffers plus forward/backward calls for one ScanWorkload.

    Inputs are taken as given (already on the device); outputs, checkpoints
    and the workspace are allocated once with torch and reused.
    """

    def __init__(self, w: W.ScanWorkload, device="cuda", want_syn: bool = False, **desc_over):
        self.w = w
        self.synaptic = w.neuron == "synaptic"
        self.recurrent = w.neuron == "rleaky"   # Eq. (7): v in the alpha slot
        self.desc = make_desc(w, **desc_over)
        self.device = torch.device(device)
        io = W.TORCH_DTYPE[w.io_dtype]
        shape = (w.T, w.B, w.N)
        dev = self.device
        self.spk = torch.empty(shape, dtype=io, device=dev)
        need_mem = w.want_mem or w.save == "mem"
        self.mem = torch.empty(shape, dtype=io, device=dev) if need_mem else None
        self.syn = torch.empty(shape, dtype=io, device=dev) if (self.synaptic and want_syn) else None
        nck = snn_scan_ckpt_elems(self.desc, self.synaptic)
        self.ckpt = torch.empty(max(nck, 1), dtype=torch.float32, device=dev) if nck > 0 else None
        self.mem_final = torch.empty((w.B, w.N), dtype=torch.float32, device=dev)
        self.syn_final = torch.empty((w.B, w.N), dtype=torch.float32, device=dev) if self.synaptic else None
        self.grad_I = torch.empty(shape, dtype=io, device=dev)
        plen = {"scalar": 1, "per_neuron": w.N, "per_channel": w.C}
        self.grad_beta = torch.empty(plen[w.beta_mode], dtype=torch.float32, device=dev)
        self.grad_thr = torch.empty(plen[w.thr_mode], dtype=torch.float32, device=dev)
        self.grad_alpha = torch.empty(plen[w.alpha_mode], dtype=torch.float32, device=dev) \
            if self.synaptic else None
        self.grad_v = torch.empty(plen[w.v_mode], dtype=torch.float32, device=dev) \
            if self.recurrent else None
        self.grad_mem0 = torch.empty((w.B, w.N), dtype=torch.float32, device=dev)
        self.grad_syn0 = torch.empty((w.B, w.N), dtype=torch.float32, device=dev) \
            if self.synaptic else None
        nws = snn_scan_workspace_bytes(self.desc)
        if nws == 0:
            raise SnnError(1, "snn_scan_workspace_bytes")
        self.ws = torch.empty(nws, dtype=torch.uint8, device=dev)
        snn_workspace_init(self.ws)

    def forward(self, I, beta, thr, alpha=None, mem0=None, syn0=None, stream=None, v=None):
        if self.recurrent:
            snn_rleaky_fwd(self.desc, I, v, beta, thr, mem0, self.spk, self.mem, self.ckpt,
                           self.mem_final, self.ws, stream)
        elif self.synaptic:
            snn_synaptic_fwd(self.desc, I, alpha, beta, thr, mem0, syn0, self.spk, self.mem,
                             self.syn, self.ckpt, self.mem_final, self.syn_final, self.ws, stream)
        else:
            snn_leaky_fwd(self.desc, I, beta, thr, mem0, self.spk, self.mem, self.ckpt,
                          self.mem_final, self.ws, stream)
        return self.spk

    def backward(self, I, beta, thr, grad_spk, alpha=None, mem0=None, syn0=None, grad_mem=None,
                 grad_mem_final=None, grad_syn_final=None, want_param_grads=True,
                 want_state_grads=True, stream=None, v=None):
        gb = self.grad_beta if want_param_grads else None
        gt = self.grad_thr if want_param_grads else None
        gm0 = self.grad_mem0 if want_state_grads else None
        recompute = self.w.save == "recompute"
        if self.recurrent:
            snn_rleaky_bwd(self.desc, I if recompute else None, self.ckpt, self.mem, self.spk, v,
                           beta, thr, mem0, grad_spk, grad_mem, grad_mem_final, self.grad_I,
                           self.grad_v if want_param_grads else None, gb, gt, gm0, self.ws,
                           stream)
        elif self.synaptic:
            ga = self.grad_alpha if (want_param_grads and (recompute or self.syn is not None)) else None
            gs0 = self.grad_syn0 if want_state_grads else None
            snn_synaptic_bwd(self.desc, I if recompute else None, self.ckpt, self.mem, self.spk,
                             self.syn, alpha, beta, thr, mem0, syn0, grad_spk, grad_mem,
                             grad_mem_final, grad_syn_final, self.grad_I, ga, gb, gt, gm0, gs0,
                             self.ws, stream)
        else:
            snn_leaky_bwd(self.desc, I if recompute else None, self.ckpt, self.mem, self.spk,
                          beta, thr, mem0, grad_spk, grad_mem, grad_mem_final, self.grad_I, gb,
                          gt, gm0, self.ws, stream)
        return self.grad_I

    def status(self, stream=None) -> int:
        return snn_workspace_status(self.ws, stream)
