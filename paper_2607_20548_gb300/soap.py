"""ctypes binding of libsoap (include/soap.h, include/muon.h): argument marshalling only.

Every step of the optimizer runs in the library's CUDA kernels; this module only
turns torch tensors into pointers and streams. It never computes anything itself,
and it raises at import if the compiled library is missing (there is no fallback).
"""
from __future__ import annotations

import ctypes
import os
import platform
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", platform.machine(), "libsoap.so")

SOAP_OK = 0
STATUS_NONFINITE, STATUS_QR_BREAKDOWN, STATUS_TIMEOUT = 1, 2, 4  # device status bits (SOAP_STATUS_*)
STATUS_NAMES = {0: "SOAP_OK", 1: "SOAP_ERR_INVALID_ARG", 2: "SOAP_ERR_CUDA", 3: "SOAP_ERR_OOM",
                4: "SOAP_ERR_NONFINITE", 5: "SOAP_ERR_QR_BREAKDOWN", 6: "SOAP_ERR_TIMEOUT"}
(STATE_M, STATE_V, STATE_L, STATE_QL, STATE_R, STATE_QR, STATE_MHAT, STATE_SKIP_L, STATE_SKIP_R,
 STATE_LAMBDA_L, STATE_LAMBDA_R) = range(11)

# every symbol include/soap.h declares
EXPORTS = ("soap_default_hparams", "soap_create", "soap_create_ex", "soap_plan_info", "soap_step", "soap_set_lr", "soap_state_bytes",
           "soap_state_get", "soap_state_set", "soap_get_step", "soap_set_step", "soap_status",
           "soap_clear_status", "soap_last_error", "soap_destroy", "soap_qr_workspace_bytes",
           "soap_qr", "soap_gemm", "soap_profile_begin", "soap_profile_begin_ex", "soap_profile_end",
           "soap_profile_records",
           "soap_gemm_tf32x4",
           "soap_split_tf32", "soap_qr_static", "soap_layerwise_assign", "soap_wait_limit")
# every symbol include/muon.h declares
MUON_EXPORTS = ("muon_default_hparams", "muon_create", "muon_step", "muon_set_lr", "muon_state_get",
                "muon_state_set", "muon_status", "muon_last_error", "muon_destroy", "muon_profile_begin",
                "muon_profile_end")
KERNEL_FAMILIES = ("gemm_simt", "gemm_tc", "qr_panel", "elementwise", "other", "qr_update")
PROFILE_SERIAL = 1  # SOAP_PROFILE_SERIAL


class muon_hparams(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("weight_decay", ctypes.c_float),
                ("eps", ctypes.c_float), ("ns_steps", ctypes.c_int32), ("coeffs", ctypes.c_void_p)]


class soap_shape(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("precond_left", ctypes.c_int32), ("precond_right", ctypes.c_int32)]


class soap_hparams(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("factor_beta", ctypes.c_float), ("eps", ctypes.c_float),
                ("weight_decay", ctypes.c_float), ("eig_every", ctypes.c_int32),
                ("bias_correction", ctypes.c_int32), ("qr_tol", ctypes.c_float),
                ("guard", ctypes.c_int32), ("kl", ctypes.c_int32),
                ("stale", ctypes.c_int32)]


class soap_kernel_stats(ctypes.Structure):
    _fields_ = [("family", ctypes.c_int32), ("launches", ctypes.c_int64), ("ms", ctypes.c_double),
                ("flops", ctypes.c_double), ("bytes", ctypes.c_double)]


class soap_launch_record(ctypes.Structure):
    _fields_ = [("family", ctypes.c_int32), ("start_ms", ctypes.c_double), ("end_ms", ctypes.c_double),
                ("flops", ctypes.c_double), ("bytes", ctypes.c_double)]


class SoapError(RuntimeError):
    def __init__(self, code, msg=""):
        super().__init__(f"{STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


_lib = None


def load_library(path: str = LIB_PATH):
    """Loads libsoap.so; raises if it has not been built (no fallback path exists)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"libsoap.so not built ({path}); run __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    P, I32, I64, F, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
    sig = {
        "soap_default_hparams": (None, [ctypes.POINTER(soap_hparams)]),
        "soap_create": (I32, [ctypes.POINTER(soap_shape), I32, ctypes.POINTER(soap_hparams), I32, ctypes.POINTER(P)]),
        "soap_create_ex": (I32, [ctypes.POINTER(soap_shape), I32, ctypes.POINTER(soap_hparams), I32, SZ,
                                 ctypes.POINTER(P)]),
        "soap_plan_info": (I32, [P, ctypes.POINTER(I32), ctypes.POINTER(I32), ctypes.POINTER(SZ),
                                 ctypes.POINTER(SZ)]),
        "soap_step": (I32, [P, P, P, P]),
        "soap_set_lr": (I32, [P, F, F]),
        "soap_state_bytes": (SZ, [P, I32, I32]),
        "soap_state_get": (I32, [P, I32, I32, P, P]),
        "soap_state_set": (I32, [P, I32, I32, P, P]),
        "soap_get_step": (I64, [P]),
        "soap_set_step": (I32, [P, I64]),
        "soap_status": (I32, [P, P]),
        "soap_clear_status": (I32, [P, P]),
        "soap_last_error": (ctypes.c_char_p, [P]),
        "soap_destroy": (None, [P]),
        "soap_qr_workspace_bytes": (SZ, [I32, I32]),
        "soap_qr": (I32, [I32, I32, P, P, P, F, P, SZ, P, P]),
        "soap_profile_begin": (I32, [P, I64]),
        "soap_profile_begin_ex": (I32, [P, I64, I32]),
        "soap_profile_end": (I32, [P, P, ctypes.POINTER(soap_kernel_stats), ctypes.POINTER(I32)]),
        "soap_profile_records": (I32, [P, ctypes.POINTER(soap_launch_record), I64, ctypes.POINTER(I64)]),
        "soap_gemm": (I32, [I32, I32, I32, I32, I32, F, P, I64, I64, P, I64, I64, F, P, I64, I64, I32, P]),
        "soap_gemm_tf32x4": (I32, [I32, I32, I32, I32, P, P, I64, I64, P, P, I64, I64, I32, F, F, P, I64, I64,
                                   I32, P, P, P]),
        "soap_split_tf32": (I32, [P, P, P, I64, P]),
        "soap_wait_limit": (I32, [ctypes.c_uint64, P]),
        "soap_qr_static": (I32, [I32, I32, P, P, P, F, P, P]),
        "soap_layerwise_assign": (I32, [ctypes.POINTER(soap_shape), I32, I32, I32, ctypes.POINTER(I32),
                                        ctypes.POINTER(ctypes.c_double)]),
        "muon_default_hparams": (None, [ctypes.POINTER(muon_hparams)]),
        "muon_create": (I32, [ctypes.POINTER(soap_shape), I32, ctypes.POINTER(muon_hparams), I32, ctypes.POINTER(P)]),
        "muon_step": (I32, [P, P, P, P]),
        "muon_set_lr": (I32, [P, F, F]),
        "muon_state_get": (I32, [P, I32, P, P]),
        "muon_state_set": (I32, [P, I32, P, P]),
        "muon_status": (I32, [P, P]),
        "muon_last_error": (ctypes.c_char_p, [P]),
        "muon_destroy": (None, [P]),
        "muon_profile_begin": (I32, [P, I64]),
        "muon_profile_end": (I32, [P, P, ctypes.POINTER(soap_kernel_stats), ctypes.POINTER(I32)]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _stream(stream=None, dev=None):
    """The cudaStream_t of `stream`, or of the current stream of device `dev` (else of the current
    device); a stream of another device than `dev` is refused before it reaches the library."""
    if dev is not None:
        dev = torch.device("cuda", dev) if isinstance(dev, int) else torch.device(dev)
    if stream is None:
        stream = torch.cuda.current_stream(dev)
    elif dev is not None and torch.device(stream.device).index != dev.index:
        raise ValueError(f"stream of {stream.device} given for work on {dev}")
    return ctypes.c_void_p(stream.cuda_stream)


def _one_device(name, *tensors, dtype=torch.float32):
    """The device the given tensors share; raises unless each is a ``dtype`` CUDA tensor on it
    (a host or a foreign-device pointer must never reach a kernel)."""
    dev = None
    for t in tensors:
        if t is None:
            continue
        if not isinstance(t, torch.Tensor) or not t.is_cuda or t.dtype != dtype:
            raise TypeError(f"{name}: expected {dtype} CUDA tensors")
        if dev is None:
            dev = t.device
        elif t.device != dev:
            raise ValueError(f"{name}: tensors on {dev} and {t.device}")
    return dev


def _check(code, h=None):
    if code != SOAP_OK:
        msg = load_library().soap_last_error(h).decode() if h else ""
        raise SoapError(code, msg)


def default_hparams(**overrides) -> soap_hparams:
    hp = soap_hparams()
    load_library().soap_default_hparams(ctypes.byref(hp))
    for k, v in overrides.items():
        setattr(hp, k, v)
    return hp


@dataclass
class Shape:
    rows: int
    cols: int
    left: bool = True
    right: bool = True


class SoapOptimizer:
    """One libsoap handle: soap_create / soap_step / soap_state_get / soap_state_set.

    workspace_limit (bytes, 0 = automatic) bounds the step's workspace (soap_create_ex): a model
    whose workspace does not fit is stepped in several waves of matrices."""

    def __init__(self, shapes, hparams: soap_hparams | None = None, device: int | None = None,
                 workspace_limit: int = 0):
        lib = load_library()
        self.shapes = [Shape(*s) if not isinstance(s, Shape) else s for s in shapes]
        arr = (soap_shape * len(self.shapes))(*[soap_shape(s.rows, s.cols, int(s.left), int(s.right))
                                               for s in self.shapes])
        self.hparams = hparams if hparams is not None else default_hparams()
        self.device = torch.cuda.current_device() if device is None else device
        h = ctypes.c_void_p()
        _check(lib.soap_create_ex(arr, len(self.shapes), ctypes.byref(self.hparams), self.device,
                                  int(workspace_limit), ctypes.byref(h)))
        self._h = h
        n = len(self.shapes)
        self._pp = (ctypes.c_void_p * n)()
        self._gp = (ctypes.c_void_p * n)()

    def _handle(self):
        if self._h is None:
            raise SoapError(1, "handle destroyed")
        return self._h

    def step(self, params, grads, stream=None):
        """soap_step on device tensors (fp32, contiguous); params are updated in place."""
        n = len(self.shapes)
        if len(params) != n or len(grads) != n:
            raise ValueError("need one param and one grad per matrix")
        for i, (p, g, s) in enumerate(zip(params, grads, self.shapes)):
            if p.dtype != torch.float32 or g.dtype != torch.float32 or not p.is_cuda or not g.is_cuda:
                raise TypeError(f"matrix {i}: params/grads must be fp32 CUDA tensors")
            if p.device.index != self.device or g.device.index != self.device:
                raise ValueError(f"matrix {i}: tensors must be on cuda:{self.device}, the handle's device")
            if tuple(p.shape) != (s.rows, s.cols) or tuple(g.shape) != (s.rows, s.cols):
                raise ValueError(f"matrix {i}: expected {(s.rows, s.cols)}")
            if not p.is_contiguous() or not g.is_contiguous():
                raise ValueError(f"matrix {i}: tensors must be contiguous")
            self._pp[i] = p.data_ptr()
            self._gp[i] = g.data_ptr()
        _check(load_library().soap_step(self._handle(), self._pp, self._gp, _stream(stream, self.device)), self._h)

    def plan_info(self) -> dict:
        """soap_plan_info: waves per step, whether they are pipelined, workspace and state bytes."""
        w, pl, ws, st = ctypes.c_int32(0), ctypes.c_int32(0), ctypes.c_size_t(0), ctypes.c_size_t(0)
        _check(load_library().soap_plan_info(self._handle(), ctypes.byref(w), ctypes.byref(pl), ctypes.byref(ws),
                                             ctypes.byref(st)), self._h)
        return {"waves": w.value, "pipelined": bool(pl.value), "workspace_bytes": ws.value, "state_bytes": st.value}

    def set_lr(self, lr: float, weight_decay: float):
        _check(load_library().soap_set_lr(self._handle(), lr, weight_decay), self._h)

    def state_bytes(self, idx: int, which: int) -> int:
        return load_library().soap_state_bytes(self._handle(), idx, which)

    def state_get(self, idx: int, which: int, stream=None) -> torch.Tensor:
        """Returns a new device tensor holding one piece of matrix idx's state."""
        s = self.shapes[idx]
        shape = {STATE_M: (s.rows, s.cols), STATE_V: (s.rows, s.cols), STATE_MHAT: (s.rows, s.cols),
                 STATE_L: (s.rows, s.rows), STATE_QL: (s.rows, s.rows), STATE_R: (s.cols, s.cols),
                 STATE_QR: (s.cols, s.cols), STATE_SKIP_L: (s.rows,), STATE_SKIP_R: (s.cols,),
                 STATE_LAMBDA_L: (s.rows,), STATE_LAMBDA_R: (s.cols,)}.get(which)
        if shape is None or self.state_bytes(idx, which) == 0:
            raise SoapError(1, f"no state piece {which} for matrix {idx}")
        dtype = torch.uint8 if which in (STATE_SKIP_L, STATE_SKIP_R) else torch.float32
        out = torch.empty(shape, dtype=dtype, device=f"cuda:{self.device}")
        _check(load_library().soap_state_get(self._handle(), idx, which, ctypes.c_void_p(out.data_ptr()),
                                             _stream(stream, self.device)), self._h)
        return out

    def state_set(self, idx: int, which: int, src: torch.Tensor, stream=None):
        if src.numel() * src.element_size() != self.state_bytes(idx, which) or not src.is_contiguous():
            raise ValueError("state_set: wrong size or non-contiguous source")
        _check(load_library().soap_state_set(self._handle(), idx, which, ctypes.c_void_p(src.data_ptr()),
                                             _stream(stream, self.device)), self._h)

    @property
    def t(self) -> int:
        return load_library().soap_get_step(self._handle())

    @t.setter
    def t(self, value: int):
        _check(load_library().soap_set_step(self._handle(), value), self._h)

    def status(self, stream=None) -> int:
        """Synchronises the stream and returns the sticky device status code."""
        return load_library().soap_status(self._handle(), _stream(stream, self.device))

    def clear_status(self, stream=None):
        _check(load_library().soap_clear_status(self._handle(), _stream(stream, self.device)), self._h)

    def profile_begin(self, max_launches: int = 1 << 16, serial: bool = False):
        """Time every kernel launch of the following calls with CUDA events; with serial, each
        launch starts on an idle device (soap_profile_begin_ex, SOAP_PROFILE_SERIAL), so its time
        is the kernel's alone."""
        _check(load_library().soap_profile_begin_ex(self._handle(), max_launches, PROFILE_SERIAL if serial else 0),
               self._h)

    def profile_end(self, stream=None) -> dict:
        """Synchronise and return {family: {launches, ms, flops, bytes}} plus an overflow flag."""
        out = (soap_kernel_stats * len(KERNEL_FAMILIES))()
        ov = ctypes.c_int32(0)
        _check(load_library().soap_profile_end(self._handle(), _stream(stream, self.device), out, ctypes.byref(ov)), self._h)
        res = {KERNEL_FAMILIES[o.family]: dict(launches=o.launches, ms=o.ms, flops=o.flops, bytes=o.bytes)
               for o in out}
        res["overflow"] = bool(ov.value)
        return res

    def profile_records(self, max_records=1 << 20, detail=False) -> list:
        """The launches timed since profile_begin as (family, start_ms, end_ms), in launch order
        (call before profile_end); with detail, (family, start_ms, end_ms, flops, bytes)."""
        out = (soap_launch_record * max_records)()
        cnt = ctypes.c_int64(0)
        _check(load_library().soap_profile_records(self._handle(), out, max_records, ctypes.byref(cnt)), self._h)
        if detail:
            return [(KERNEL_FAMILIES[out[i].family], out[i].start_ms, out[i].end_ms, out[i].flops, out[i].bytes)
                    for i in range(cnt.value)]
        return [(KERNEL_FAMILIES[out[i].family], out[i].start_ms, out[i].end_ms) for i in range(cnt.value)]

    def last_error(self) -> str:
        return load_library().soap_last_error(self._handle()).decode()

    def destroy(self):
        if self._h is not None:
            load_library().soap_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


# ---- module-level names matching the C ABI ------------------------------------------

def soap_create(shapes, hparams=None, device=None) -> SoapOptimizer:
    return SoapOptimizer(shapes, hparams, device)


def soap_step(opt: SoapOptimizer, params, grads, stream=None):
    opt.step(params, grads, stream)


def soap_state_get(opt: SoapOptimizer, idx, which, stream=None):
    return opt.state_get(idx, which, stream)


def soap_state_set(opt: SoapOptimizer, idx, which, src, stream=None):
    opt.state_set(idx, which, src, stream)


def soap_qr(P: torch.Tensor, tol: float = 0.0, stream=None, return_status=False):
    """Batched QR refresh on device: P [batch, n, n] fp32 -> (Q, skip[batch, n] uint8), and with
    return_status the call's device status word (an int32 tensor: 0, or SOAP_STATUS_* bits)."""
    lib = load_library()
    if P.dim() == 2:
        P = P.unsqueeze(0)
    if P.dtype != torch.float32 or not P.is_cuda or P.shape[1] != P.shape[2]:
        raise TypeError("soap_qr: P must be a [batch, n, n] fp32 CUDA tensor")
    P = P.contiguous()
    batch, n = P.shape[0], P.shape[1]
    Q = torch.empty_like(P)
    skip = torch.empty(batch, n, dtype=torch.uint8, device=P.device)
    ws_bytes = lib.soap_qr_workspace_bytes(n, batch)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=P.device)
    status = torch.empty(1, dtype=torch.int32, device=P.device)
    with torch.cuda.device(P.device):
        _check(lib.soap_qr(n, batch, ctypes.c_void_p(P.data_ptr()), ctypes.c_void_p(Q.data_ptr()),
                           ctypes.c_void_p(skip.data_ptr()), float(tol), ctypes.c_void_p(ws.data_ptr()), ws_bytes,
                           ctypes.c_void_p(status.data_ptr()), _stream(stream, P.device)))
    return (Q, skip, status) if return_status else (Q, skip)


def soap_qr_static(P: torch.Tensor, tol: float = 0.0, stream=None, return_status=False):
    """soap_qr without a caller-supplied workspace, for code that cannot allocate device memory
    when it needs the QR: libsoap.so uses a fixed 32 MiB array of its own (enough for one
    1024 x 1024 matrix). The output tensors here are allocated by torch for convenience; a
    caller without an allocator passes its own buffers to the C entry point. Raises
    SoapError(SOAP_ERR_INVALID_ARG) for work larger than the array. With return_status, also
    returns the call's device status word (an int32 tensor: 0, or SOAP_STATUS_* bits)."""
    lib = load_library()
    if P.dim() == 2:
        P = P.unsqueeze(0)
    if P.dtype != torch.float32 or not P.is_cuda or P.shape[1] != P.shape[2]:
        raise TypeError("soap_qr_static: P must be a [batch, n, n] fp32 CUDA tensor")
    P = P.contiguous()
    batch, n = P.shape[0], P.shape[1]
    Q = torch.empty_like(P)
    skip = torch.empty(batch, n, dtype=torch.uint8, device=P.device)
    status = torch.empty(1, dtype=torch.int32, device=P.device)
    with torch.cuda.device(P.device):
        code = lib.soap_qr_static(n, batch, ctypes.c_void_p(P.data_ptr()), ctypes.c_void_p(Q.data_ptr()),
                                  ctypes.c_void_p(skip.data_ptr()), float(tol), ctypes.c_void_p(status.data_ptr()),
                                  _stream(stream, P.device))
    if code != SOAP_OK:
        raise SoapError(code, f"soap_qr_static(n={n}, batch={batch}): needs "
                              f"{lib.soap_qr_workspace_bytes(n, batch)} bytes of workspace; the fixed array "
                              "holds 32 MiB" if code == 1 else "soap_qr_static failed")
    return (Q, skip, status) if return_status else (Q, skip)


def soap_wait_limit(limit_ns: int = 0, hold: torch.Tensor | None = None):
    """soap_wait_limit: bound of the tensor-core products' device waits (0 = default 2 s) and an
    optional int32 CUDA flag their epilogues first wait for (testing the timeout path)."""
    if hold is not None:
        _one_device("soap_wait_limit hold", hold, dtype=torch.int32)
    _check(load_library().soap_wait_limit(int(limit_ns), ctypes.c_void_p(hold.data_ptr()) if hold is not None else None))


def soap_gemm(A: torch.Tensor, B: torch.Tensor, trans_a=False, trans_b=False, alpha=1.0, beta=0.0,
              C: torch.Tensor | None = None, stream=None):
    """C = alpha op(A) op(B) + beta C on [batch, r, c] (or 2-D) fp32 CUDA tensors."""
    lib = load_library()
    squeeze = A.dim() == 2
    A3 = (A.unsqueeze(0) if A.dim() == 2 else A).contiguous()
    B3 = (B.unsqueeze(0) if B.dim() == 2 else B).contiguous()
    batch = A3.shape[0]
    M = A3.shape[2] if trans_a else A3.shape[1]
    K = A3.shape[1] if trans_a else A3.shape[2]
    N = B3.shape[1] if trans_b else B3.shape[2]
    dev = _one_device("soap_gemm", A3, B3, C)
    if C is None:
        C3 = torch.zeros(batch, M, N, dtype=torch.float32, device=dev)
    else:
        C3 = C.unsqueeze(0) if C.dim() == 2 else C
        if not C3.is_contiguous():
            raise ValueError("C must be contiguous")
    with torch.cuda.device(dev):
        _check(lib.soap_gemm(int(trans_a), int(trans_b), M, N, K, float(alpha),
                             ctypes.c_void_p(A3.data_ptr()), A3.shape[2], A3.shape[1] * A3.shape[2],
                             ctypes.c_void_p(B3.data_ptr()), B3.shape[2], B3.shape[1] * B3.shape[2], float(beta),
                             ctypes.c_void_p(C3.data_ptr()), N, M * N, batch, _stream(stream, dev)))
    return C3[0] if squeeze else C3


def soap_split_tf32(x: torch.Tensor, stream=None):
    """(hi, lo) with hi = x truncated to tf32 and lo = x - hi, computed on the device."""
    dev = _one_device("soap_split_tf32", x)
    x = x.contiguous()
    hi, lo = torch.empty_like(x), torch.empty_like(x)
    with torch.cuda.device(dev):
        _check(load_library().soap_split_tf32(ctypes.c_void_p(x.data_ptr()), ctypes.c_void_p(hi.data_ptr()),
                                              ctypes.c_void_p(lo.data_ptr()), x.numel(), _stream(stream, dev)))
    return hi, lo


def soap_gemm_tf32x4(A, B, alpha=1.0, beta=0.0, C=None, transpose_c=False, A_split=None, B_split=None,
                     with_lo=False, status=None, stream=None):
    """Tensor-core C = alpha A B^T + beta C for [batch, M, K] x [b_batch, N, K] fp32 CUDA tensors.

    A_split / B_split give (hi, lo) explicitly; by default they come from soap_split_tf32.
    Returns C (and C_lo if with_lo)."""
    lib = load_library()
    A3 = (A.unsqueeze(0) if A.dim() == 2 else A).contiguous()
    B3 = (B.unsqueeze(0) if B.dim() == 2 else B).contiguous()
    batch, M, K = A3.shape
    bb, N, K2 = B3.shape
    if K != K2:
        raise ValueError("soap_gemm_tf32x4: A and B need the same K")
    dev = _one_device("soap_gemm_tf32x4", A3, B3, C)
    if status is not None:
        _one_device("soap_gemm_tf32x4 status", status, dtype=torch.int32)
        if status.device != dev:
            raise ValueError("soap_gemm_tf32x4: status on another device")
    ahi, alo = A_split if A_split is not None else soap_split_tf32(A3, stream)
    bhi, blo = B_split if B_split is not None else soap_split_tf32(B3, stream)
    if _one_device("soap_gemm_tf32x4 splits", ahi, alo, bhi, blo) != dev:
        raise ValueError("soap_gemm_tf32x4: split operands on another device")
    shape = (batch, N, M) if transpose_c else (batch, M, N)
    C3 = torch.zeros(shape, dtype=torch.float32, device=A3.device) if C is None else \
        (C.unsqueeze(0) if C.dim() == 2 else C)
    lo = torch.zeros_like(C3) if with_lo else None
    ldc = shape[2]
    with torch.cuda.device(dev):
        _check(lib.soap_gemm_tf32x4(M, N, K, batch, ctypes.c_void_p(ahi.data_ptr()), ctypes.c_void_p(alo.data_ptr()),
                                    K, M * K, ctypes.c_void_p(bhi.data_ptr()), ctypes.c_void_p(blo.data_ptr()), K,
                                    N * K, bb, float(alpha), float(beta), ctypes.c_void_p(C3.data_ptr()), ldc,
                                    shape[1] * shape[2], int(transpose_c),
                                    ctypes.c_void_p(lo.data_ptr()) if with_lo else None,
                                    ctypes.c_void_p(status.data_ptr()) if status is not None else None,
                                    _stream(stream, dev)))
    out = C3[0] if A.dim() == 2 and (C is None or C.dim() == 2) else C3
    if with_lo:
        return out, (lo[0] if out.dim() == 2 else lo)
    return out


class MuonOptimizer:
    """One Muon handle (include/muon.h): muon_create / muon_step / muon_state_get / set.

    ``coeffs`` is a list of (a_i, b_i, c_i) Newton-Schulz coefficients (None: the library's
    default quintic schedule); its length sets the number of iterations."""

    def __init__(self, shapes, lr=3e-3, beta1=0.9, weight_decay=0.1, eps=1e-7, coeffs=None, ns_steps=16,
                 device: int | None = None):
        lib = load_library()
        self.shapes = [(int(s[0]), int(s[1])) for s in shapes]
        arr = (soap_shape * len(self.shapes))(*[soap_shape(r, c, 0, 0) for r, c in self.shapes])
        hp = muon_hparams()
        lib.muon_default_hparams(ctypes.byref(hp))
        hp.lr, hp.beta1, hp.weight_decay, hp.eps = lr, beta1, weight_decay, eps
        self._coeffs = None
        if coeffs is not None:
            flat = [float(x) for abc in coeffs for x in abc]
            self._coeffs = (ctypes.c_float * len(flat))(*flat)
            hp.ns_steps = len(coeffs)
            hp.coeffs = ctypes.cast(self._coeffs, ctypes.c_void_p)
        else:
            hp.ns_steps = ns_steps
        self.device = torch.cuda.current_device() if device is None else device
        h = ctypes.c_void_p()
        code = lib.muon_create(arr, len(self.shapes), ctypes.byref(hp), self.device, ctypes.byref(h))
        if code != SOAP_OK:
            raise SoapError(code, "muon_create")
        self._h = h
        n = len(self.shapes)
        self._pp = (ctypes.c_void_p * n)()
        self._gp = (ctypes.c_void_p * n)()

    def _handle(self):
        if self._h is None:
            raise SoapError(1, "handle destroyed")
        return self._h

    def _check(self, code):
        if code != SOAP_OK:
            raise SoapError(code, load_library().muon_last_error(self._h).decode())

    def step(self, params, grads, stream=None):
        """muon_step on device tensors (fp32, contiguous); params are updated in place."""
        n = len(self.shapes)
        if len(params) != n or len(grads) != n:
            raise ValueError("need one param and one grad per matrix")
        for i, (p, g, s) in enumerate(zip(params, grads, self.shapes)):
            if p.dtype != torch.float32 or g.dtype != torch.float32 or not p.is_cuda or not g.is_cuda:
                raise TypeError(f"matrix {i}: params/grads must be fp32 CUDA tensors")
            if p.device.index != self.device or g.device.index != self.device:
                raise ValueError(f"matrix {i}: tensors must be on cuda:{self.device}, the handle's device")
            if tuple(p.shape) != s or tuple(g.shape) != s or not p.is_contiguous() or not g.is_contiguous():
                raise ValueError(f"matrix {i}: expected a contiguous {s} tensor")
            self._pp[i] = p.data_ptr()
            self._gp[i] = g.data_ptr()
        self._check(load_library().muon_step(self._handle(), self._pp, self._gp, _stream(stream, self.device)))

    def set_lr(self, lr: float, weight_decay: float):
        self._check(load_library().muon_set_lr(self._handle(), lr, weight_decay))

    def state_get(self, idx: int, stream=None) -> torch.Tensor:
        """The momentum M of matrix idx as a new device tensor."""
        out = torch.empty(self.shapes[idx], dtype=torch.float32, device=f"cuda:{self.device}")
        self._check(load_library().muon_state_get(self._handle(), idx, ctypes.c_void_p(out.data_ptr()),
                                                  _stream(stream, self.device)))
        return out

    def state_set(self, idx: int, src: torch.Tensor, stream=None):
        if tuple(src.shape) != self.shapes[idx] or src.dtype != torch.float32 or not src.is_contiguous():
            raise ValueError("state_set: wrong shape, dtype or layout")
        self._check(load_library().muon_state_set(self._handle(), idx, ctypes.c_void_p(src.data_ptr()),
                                                  _stream(stream, self.device)))

    def status(self, stream=None) -> int:
        return load_library().muon_status(self._handle(), _stream(stream, self.device))

    def last_error(self) -> str:
        return load_library().muon_last_error(self._h).decode() if self._h else "handle destroyed"

    def profile_begin(self, max_launches: int = 1 << 16):
        """Time every kernel launch of the following calls with CUDA events."""
        self._check(load_library().muon_profile_begin(self._handle(), max_launches))

    def profile_end(self, stream=None) -> dict:
        """Synchronise and return {family: {launches, ms, flops, bytes}} plus an overflow flag."""
        out = (soap_kernel_stats * len(KERNEL_FAMILIES))()
        ov = ctypes.c_int32(0)
        self._check(load_library().muon_profile_end(self._handle(), _stream(stream, self.device), out, ctypes.byref(ov)))
        res = {KERNEL_FAMILIES[o.family]: dict(launches=o.launches, ms=o.ms, flops=o.flops, bytes=o.bytes)
               for o in out}
        res["overflow"] = bool(ov.value)
        return res

    def destroy(self):
        if self._h is not None:
            load_library().muon_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def layerwise_assign(shapes, world: int, policy: int = 0):
    """soap_layerwise_assign: (owner per matrix, cost per rank) for `world` ranks."""
    n = len(shapes)
    arr = (soap_shape * n)(*[soap_shape(int(s[0]), int(s[1]), int(s[2]) if len(s) > 2 else 1,
                                        int(s[3]) if len(s) > 3 else 1) for s in shapes])
    owner = (ctypes.c_int32 * n)()
    load = (ctypes.c_double * world)()
    code = load_library().soap_layerwise_assign(arr, n, world, policy, owner, load)
    if code != SOAP_OK:
        raise SoapError(code, "soap_layerwise_assign")
    return list(owner), list(load)
