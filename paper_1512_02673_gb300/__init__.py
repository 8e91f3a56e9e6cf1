"""Python binding of libcm (MDS-coded matrix multiplication on one GB300).

Thin ctypes marshalling over the C ABI declared in ``include/cm.h``: every
function here checks tensor dtypes, devices and shapes, passes raw pointers
and the current torch CUDA stream, and maps status codes to exceptions.  All
computation runs in the library's CUDA kernels; there is no fallback, and
importing a function whose library was not built raises ``LibraryMissing``.

Method: Lee et al., "Speeding Up Distributed Machine Learning Using Codes",
Sec. III (see ``include/cm.h`` for the definitions of each call).
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libcm.so")

CM_OK, CM_EINVAL, CM_ENOTDECODABLE, CM_ESINGULAR = 0, -1, -2, -3
CM_ECUDA, CM_ENOMEM, CM_ETIMEOUT, CM_EUNSUPPORTED = -4, -5, -6, -7
CM_F32, CM_BF16 = 0, 1


class LibraryMissing(RuntimeError):
    pass


class CodedError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__("%s: %s (status %d)" % (what, status_string(status), status))


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libcm (raises LibraryMissing if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise LibraryMissing("libcm.so is not built: run "
                                 "`python -m paper_1512_02673_gb300.build`")
        L = ctypes.CDLL(LIB_PATH)
        i32, i64, u32, u64, f32, f64 = (ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32,
                                        ctypes.c_uint64, ctypes.c_float, ctypes.c_double)
        vp, sz = ctypes.c_void_p, ctypes.c_size_t
        st = ctypes.c_int
        sig = {
            "cm_code_create": (st, [i32, i32, i64, i64, st, vp, ctypes.POINTER(vp)]),
            "cm_code_destroy": (None, [vp]),
            "cm_block_rows": (i64, [vp]),
            "cm_encode": (st, [vp, vp, i64, vp, i64, vp, vp]),
            "cm_matvec": (st, [vp, vp, i64, vp, i64, vp, i32, vp, vp, vp]),
            "cm_matvec_survivors": (st, [vp, vp, i64, vp, i64, vp, i32, u32, vp, vp, vp]),
            "cm_draw_erasures": (st, [u64, u64, i32, i32, f64, f64, ctypes.POINTER(u32), vp]),
            "cm_decode": (st, [vp, vp, u32, i32, vp, vp, vp]),
            "cm_gd_workspace_bytes": (sz, [vp, vp]),
            "cm_matvec_decode_workspace_bytes": (sz, [vp, i32]),
            "cm_matvec_decode": (st, [vp, vp, i64, vp, i64, vp, i32, u32, i32, vp, vp, sz, vp,
                                      vp]),
            "cm_gd_step_survivors": (st, [vp, vp, i64, vp, i64, vp, vp, i64, vp, i64, vp, vp, f32,
                                          u32, u32, vp, sz, vp, vp]),
            "cm_gd_step": (st, [vp, vp, i64, vp, i64, vp, vp, i64, vp, i64, vp, vp, f32,
                                u32, u32, vp, sz, vp, vp]),
            "cm_gd_step_noalloc": (st, [vp, vp, i64, vp, i64, vp, vp, i64, vp, i64, vp, vp,
                                        f32, u32, u32, vp, vp]),
            "cm_coded_gemm": (st, [vp, vp, i64, vp, i64, vp, i64, i32, vp, i64, vp, vp]),
            "cm_coded_gemm_survivors": (st, [vp, vp, i64, vp, i64, vp, i64, i32, u32, vp,
                                             i64, vp, vp]),
            "cm_decode_mat": (st, [vp, vp, i64, u32, i32, vp, i64, vp, vp]),
            "cm_matmat": (st, [vp, vp, i64, vp, i64, vp, i64, i32, vp, i64, u32, vp, i64,
                               vp, vp]),
            "cm_selftest_bounded_wait": (st, [vp, u64, vp]),
            "cm_status_string": (ctypes.c_char_p, [st]),
            "cm_code_create_repetition": (st, [i32, i32, i64, i64, st, ctypes.POINTER(vp)]),
            "cm_select_decodable": (st, [vp, u32, ctypes.POINTER(u32)]),
            "cm_runtime_mean": (st, [st, i32, i32, f64, f64, ctypes.POINTER(f64)]),
            "cm_runtime_cdf": (st, [st, i32, i32, f64, f64, vp, i64, vp]),
            "cm_runtime_simulate": (st, [st, i32, i32, f64, f64, u64, u64, i64, vp]),
            "cm_optimal_mds_k": (st, [i32, f64, ctypes.POINTER(f64), ctypes.POINTER(f64)]),
            "cm_shuffle_create": (st, [i32, i64, i64, u64, u64, ctypes.POINTER(vp)]),
            "cm_shuffle_destroy": (None, [vp]),
            "cm_shuffle_next": (st, [vp, vp]),
            "cm_shuffle_query": (st, [vp, vp]),
            "cm_shuffle_plan": (st, [vp, vp, vp, vp, vp]),
            "cm_shuffle_received": (st, [vp, vp, vp]),
            "cm_shuffle_caches": (st, [vp, vp, vp]),
            "cm_shuffle_rates": (st, [i32, f64, f64, ctypes.POINTER(f64), ctypes.POINTER(f64)]),
            "cm_shuffle_workspace_bytes": (sz, [vp]),
            "cm_shuffle_upload": (st, [vp, vp, sz, vp]),
            "cm_shuffle_fill": (st, [vp, vp, vp, i64, i64, vp, i64, vp]),
            "cm_shuffle_encode": (st, [vp, vp, st, vp, i64, i64, vp, i64, vp]),
            "cm_shuffle_decode": (st, [vp, vp, st, vp, i64, vp, i64, i64, vp, i64, vp]),
            "cm_shuffle_commit": (st, [vp, vp, vp, i64, i64, vp, i64, vp]),
            "cm_shuffle_device_workspace_bytes": (sz, [vp]),
            "cm_shuffle_device_init": (st, [vp, vp, sz, vp]),
            "cm_shuffle_device_next": (st, [vp, vp, sz, vp, vp]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().cm_status_string(status).decode()


def _check(status: int, what: str):
    if status != CM_OK:
        raise CodedError(status, what)


# The current CUDA stream of the current device as a raw handle.  torch's
# internal accessors return it in well under a microsecond, against a few
# microseconds for torch.cuda.current_stream() (a Python stream object per
# call); the public call stays as the fallback.
_raw_stream = getattr(torch._C, "_cuda_getCurrentRawStream", None)
_cur_device = getattr(torch._C, "_cuda_getDevice", None)


def _stream():
    if _raw_stream is not None and _cur_device is not None:
        return _raw_stream(_cur_device())
    return torch.cuda.current_stream().cuda_stream


def _dev(t: torch.Tensor, dtype, name: str, ndim=None) -> int:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError("%s must be a CUDA tensor" % name)
    if t.dtype != dtype:
        raise TypeError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if ndim is not None and t.dim() != ndim:
        raise ValueError("%s must have %d dimensions" % (name, ndim))
    return t.data_ptr()


def _ld(t: torch.Tensor, name: str) -> int:
    """Leading dimension of a row-major matrix view (unit column stride)."""
    if t.dim() != 2 or (t.shape[1] > 1 and t.stride(1) != 1):
        raise ValueError("%s must be a row-major matrix" % name)
    return t.stride(0)


def _contig(t: torch.Tensor, name: str):
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)


class Code:
    """An (n,k) systematic code G = [I_k; P] for an m x d data matrix.

    parity="repetition" builds the n/k-repetition code (worker j holds block
    j mod k); otherwise parity is the (n-k) x k block P."""

    def __init__(self, n: int, k: int, m: int, d: int, parity, dtype: str = "f32"):
        dt = {"f32": CM_F32, "bf16": CM_BF16}[dtype]
        out = ctypes.c_void_p()
        if isinstance(parity, str) and parity == "repetition":
            _check(lib().cm_code_create_repetition(n, k, m, d, dt, ctypes.byref(out)),
                   "cm_code_create_repetition")
            P = np.zeros((n - k, k), np.float32)
            for p in range(n - k):
                P[p, p % k] = 1.0
        else:
            P = np.ascontiguousarray(np.asarray(parity, dtype=np.float32))
            if P.shape != (n - k, k):
                raise ValueError("parity must be (n-k) x k")
            _check(lib().cm_code_create(n, k, m, d, dt, P.ctypes.data_as(ctypes.c_void_p),
                                        ctypes.byref(out)), "cm_code_create")
        self._h = out
        self.n, self.k, self.m, self.d, self.dtype = n, k, m, d, dtype
        self.P = P
        self.L = int(lib().cm_block_rows(out))

    @property
    def handle(self):
        return self._h

    def select_decodable(self, survivors: int) -> int:
        """The k workers a decode uses for this survivor mask (bitmask)."""
        sel = ctypes.c_uint32(0)
        _check(lib().cm_select_decodable(self._h, survivors, ctypes.byref(sel)),
               "cm_select_decodable")
        return int(sel.value)

    def __del__(self):
        h = getattr(self, "_h", None)
        if h and _lib is not None:
            _lib.cm_code_destroy(h)
            self._h = None

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16


def encode(code: Code, A: torch.Tensor, parity: torch.Tensor | None = None,
           status: torch.Tensor | None = None) -> torch.Tensor:
    """Parity blocks ((n-k) L x d, code dtype) of A (m x d)."""
    dt = code.torch_dtype
    _dev(A, dt, "A", 2)
    if tuple(A.shape) != (code.m, code.d):
        raise ValueError("A must be m x d")
    if parity is None:
        # rows start on 16-byte boundaries (the library's layout contract)
        per16 = 16 // A.element_size()
        ldp = (code.d + per16 - 1) // per16 * per16
        parity = torch.empty(((code.n - code.k) * code.L, ldp), dtype=dt,
                             device=A.device)[:, :code.d]
    _dev(parity, dt, "parity", 2)
    if tuple(parity.shape) != ((code.n - code.k) * code.L, code.d):
        raise ValueError("parity must be (n-k) L x d")
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_encode(code.handle, A.data_ptr(), _ld(A, "A"), parity.data_ptr(),
                           _ld(parity, "parity"), sp, _stream()), "cm_encode")
    return parity


def matvec(code: Code, A: torch.Tensor, parity: torch.Tensor, X: torch.Tensor,
           Yt: torch.Tensor | None = None, status: torch.Tensor | None = None) -> torch.Tensor:
    """All n worker products Yt (n L x b, fp64) for X (d x b fp32, b <= 8)."""
    _dev(A, torch.float32, "A", 2)
    _dev(parity, torch.float32, "parity", 2)
    if X.dim() == 1:
        X = X.view(-1, 1)
    _dev(X, torch.float32, "X", 2)
    _contig(X, "X")
    if X.shape[0] != code.d:
        raise ValueError("X must have d rows")
    b = X.shape[1]
    if Yt is None:
        Yt = torch.empty((code.n * code.L, b), dtype=torch.float64, device=X.device)
    _dev(Yt, torch.float64, "Yt", 2)
    _contig(Yt, "Yt")
    if tuple(Yt.shape) != (code.n * code.L, b):
        raise ValueError("Yt must be n L x b")
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_matvec(code.handle, A.data_ptr(), _ld(A, "A"), parity.data_ptr(),
                           _ld(parity, "parity"), X.data_ptr(), b, Yt.data_ptr(), sp,
                           _stream()), "cm_matvec")
    return Yt


def matvec_survivors(code: Code, A: torch.Tensor, parity: torch.Tensor, X: torch.Tensor,
                     survivors: int, Yt: torch.Tensor | None = None,
                     status: torch.Tensor | None = None) -> torch.Tensor:
    """Worker products of the k survivors only (the other rows of Yt untouched)."""
    _dev(A, torch.float32, "A", 2)
    _dev(parity, torch.float32, "parity", 2)
    if X.dim() == 1:
        X = X.view(-1, 1)
    _dev(X, torch.float32, "X", 2)
    _contig(X, "X")
    b = X.shape[1]
    if Yt is None:
        Yt = torch.empty((code.n * code.L, b), dtype=torch.float64, device=X.device)
    _dev(Yt, torch.float64, "Yt", 2)
    _contig(Yt, "Yt")
    if tuple(Yt.shape) != (code.n * code.L, b) or X.shape[0] != code.d:
        raise ValueError("shapes: X must be d x b and Yt n L x b")
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_matvec_survivors(code.handle, A.data_ptr(), _ld(A, "A"), parity.data_ptr(),
                                     _ld(parity, "parity"), X.data_ptr(), b, survivors,
                                     Yt.data_ptr(), sp, _stream()), "cm_matvec_survivors")
    return Yt


def draw_erasures(seed: int, counter: int, n: int, k: int, shift: float = 1.0,
                  rate: float = 1.0):
    """(survivor bitmask, n task times) of one shifted-exponential straggler draw."""
    mask = ctypes.c_uint32(0)
    times = np.empty(n, np.float64)
    _check(lib().cm_draw_erasures(seed, counter, n, k, shift, rate, ctypes.byref(mask),
                                  times.ctypes.data_as(ctypes.c_void_p)), "cm_draw_erasures")
    return int(mask.value), times


def decode(code: Code, Yt: torch.Tensor, survivors: int, Y: torch.Tensor | None = None,
           status: torch.Tensor | None = None) -> torch.Tensor:
    """Y = A X (m x b fp32) decoded from the surviving rows of Yt."""
    _dev(Yt, torch.float64, "Yt", 2)
    _contig(Yt, "Yt")
    b = Yt.shape[1]
    if Y is None:
        Y = torch.empty((code.m, b), dtype=torch.float32, device=Yt.device)
    _dev(Y, torch.float32, "Y", 2)
    _contig(Y, "Y")
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_decode(code.handle, Yt.data_ptr(), survivors, b, Y.data_ptr(), sp,
                           _stream()), "cm_decode")
    return Y


def gd_workspace_bytes(code_A: Code, code_AT: Code) -> int:
    return int(lib().cm_gd_workspace_bytes(code_A.handle, code_AT.handle))


def matvec_decode_workspace_bytes(code: Code, b: int) -> int:
    return int(lib().cm_matvec_decode_workspace_bytes(code.handle, b))


def matvec_decode(code: Code, A: torch.Tensor, parity: torch.Tensor, X: torch.Tensor,
                  survivors: int, only_survivors: bool = False, Y: torch.Tensor | None = None,
                  ws: torch.Tensor | None = None,
                  status: torch.Tensor | None = None) -> torch.Tensor:
    """Y = A X (m x b fp32): the worker products with the decode fused into
    their tail.  only_survivors computes only the k used workers.  ws (uint8,
    at least matvec_decode_workspace_bytes) also holds the stacked results;
    allocated here when not given."""
    _dev(A, torch.float32, "A", 2)
    _dev(parity, torch.float32, "parity", 2)
    if X.dim() == 1:
        X = X.view(-1, 1)
    _dev(X, torch.float32, "X", 2)
    _contig(X, "X")
    if X.shape[0] != code.d:
        raise ValueError("X must have d rows")
    b = X.shape[1]
    if Y is None:
        Y = torch.empty((code.m, b), dtype=torch.float32, device=X.device)
    _dev(Y, torch.float32, "Y", 2)
    _contig(Y, "Y")
    if ws is None:
        ws = torch.empty(matvec_decode_workspace_bytes(code, b), dtype=torch.uint8,
                         device=X.device)
    _dev(ws, torch.uint8, "ws")
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_matvec_decode(code.handle, A.data_ptr(), _ld(A, "A"), parity.data_ptr(),
                                  _ld(parity, "parity"), X.data_ptr(), b, survivors,
                                  1 if only_survivors else 0, Y.data_ptr(), ws.data_ptr(),
                                  ws.numel(), sp, _stream()), "cm_matvec_decode")
    return Y


def gd_step(code_A: Code, A, PA, code_AT: Code, AT, PAT, y, x, eta: float, surv_A: int,
            surv_AT: int, ws: torch.Tensor, status: torch.Tensor | None = None,
            survivors_only: bool = False):
    """One coded gradient step x <- x - eta A^T (A x - y), x updated in place.
    survivors_only computes only the k used workers of each product."""
    for t, name in ((A, "A"), (PA, "PA"), (AT, "AT"), (PAT, "PAT")):
        _dev(t, torch.float32, name, 2)
    _dev(y, torch.float32, "y")
    _dev(x, torch.float32, "x")
    _contig(x, "x")
    _contig(y, "y")
    _dev(ws, torch.uint8, "ws")
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    fn = lib().cm_gd_step_survivors if survivors_only else lib().cm_gd_step
    _check(fn(code_A.handle, A.data_ptr(), _ld(A, "A"), PA.data_ptr(), _ld(PA, "PA"),
              code_AT.handle, AT.data_ptr(), _ld(AT, "AT"), PAT.data_ptr(), _ld(PAT, "PAT"),
              y.data_ptr(), x.data_ptr(), eta, surv_A, surv_AT, ws.data_ptr(), ws.numel(), sp,
              _stream()), "cm_gd_step_survivors" if survivors_only else "cm_gd_step")
    return x


# Size of the fixed device scratch array behind gd_step_noalloc (bytes).
GD_STATIC_SCRATCH_BYTES = 4 << 20


def gd_step_noalloc(code_A: Code, A, PA, code_AT: Code, AT, PAT, y, x, eta: float,
                    surv_A: int, surv_AT: int, status: torch.Tensor | None = None):
    """gd_step for callers that cannot allocate device memory.

    Uses the library's fixed device scratch array (GD_STATIC_SCRATCH_BYTES,
    shared by all calls on a device) instead of a workspace argument, and
    allocates nothing.  Problems whose workspace would exceed the array raise
    CodedError(CM_ENOMEM).  Calls that overlap on the GPU race on the array."""
    for t, name in ((A, "A"), (PA, "PA"), (AT, "AT"), (PAT, "PAT")):
        _dev(t, torch.float32, name, 2)
    _dev(y, torch.float32, "y")
    _dev(x, torch.float32, "x")
    _contig(x, "x")
    _contig(y, "y")
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_gd_step_noalloc(code_A.handle, A.data_ptr(), _ld(A, "A"), PA.data_ptr(),
                                    _ld(PA, "PA"), code_AT.handle, AT.data_ptr(),
                                    _ld(AT, "AT"), PAT.data_ptr(), _ld(PAT, "PAT"),
                                    y.data_ptr(), x.data_ptr(), eta, surv_A, surv_AT, sp,
                                    _stream()), "cm_gd_step_noalloc")
    return x


def selftest_bounded_wait(status: torch.Tensor, limit_ns: int) -> None:
    """Run the library's bounded-wait self-test: a device wait that nothing
    completes must give up after limit_ns and write CM_ETIMEOUT to status."""
    _dev(status, torch.int32, "status")
    _check(lib().cm_selftest_bounded_wait(status.data_ptr(), limit_ns, _stream()),
           "cm_selftest_bounded_wait")


def coded_gemm(code: Code, A, parity, Bt, Ct=None, status=None) -> torch.Tensor:
    """All n worker products Ct = A~ B (n L x N fp32) on tensor cores.

    Bt is B transposed: N x d bf16 (each column of B contiguous)."""
    for t, name in ((A, "A"), (parity, "parity"), (Bt, "Bt")):
        _dev(t, torch.bfloat16, name, 2)
    N = Bt.shape[0]
    if Ct is None:
        Ct = torch.empty((code.n * code.L, N), dtype=torch.float32, device=A.device)
    _dev(Ct, torch.float32, "Ct", 2)
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_coded_gemm(code.handle, A.data_ptr(), _ld(A, "A"), parity.data_ptr(),
                               _ld(parity, "parity"), Bt.data_ptr(), _ld(Bt, "Bt"), N,
                               Ct.data_ptr(), _ld(Ct, "Ct"), sp, _stream()), "cm_coded_gemm")
    return Ct


def coded_gemm_survivors(code: Code, A, parity, Bt, survivors: int, Ct=None,
                         status=None) -> torch.Tensor:
    """Worker products of the k workers decode_mat reads (the other blocks of Ct
    untouched)."""
    for t, name in ((A, "A"), (parity, "parity"), (Bt, "Bt")):
        _dev(t, torch.bfloat16, name, 2)
    N = Bt.shape[0]
    if Ct is None:
        Ct = torch.empty((code.n * code.L, N), dtype=torch.float32, device=A.device)
    _dev(Ct, torch.float32, "Ct", 2)
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_coded_gemm_survivors(code.handle, A.data_ptr(), _ld(A, "A"),
                                         parity.data_ptr(), _ld(parity, "parity"),
                                         Bt.data_ptr(), _ld(Bt, "Bt"), N, survivors,
                                         Ct.data_ptr(), _ld(Ct, "Ct"), sp, _stream()),
           "cm_coded_gemm_survivors")
    return Ct


def decode_mat(code: Code, Ct: torch.Tensor, survivors: int, C: torch.Tensor | None = None,
               status: torch.Tensor | None = None) -> torch.Tensor:
    """C = A B (m x N fp32) decoded from the surviving blocks of Ct (may alias Ct)."""
    _dev(Ct, torch.float32, "Ct", 2)
    N = Ct.shape[1]
    if C is None:
        C = torch.empty((code.m, N), dtype=torch.float32, device=Ct.device)
    _dev(C, torch.float32, "C", 2)
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_decode_mat(code.handle, Ct.data_ptr(), _ld(Ct, "Ct"), survivors, N,
                               C.data_ptr(), _ld(C, "C"), sp, _stream()), "cm_decode_mat")
    return C


def matmat(code: Code, A, parity, Bt, survivors: int, Ct=None, C=None, status=None):
    """(Ct, C): coded GEMM of all n workers, then decode from the survivors."""
    for t, name in ((A, "A"), (parity, "parity"), (Bt, "Bt")):
        _dev(t, torch.bfloat16, name, 2)
    N = Bt.shape[0]
    if Ct is None:
        Ct = torch.empty((code.n * code.L, N), dtype=torch.float32, device=A.device)
    if C is None:
        C = torch.empty((code.m, N), dtype=torch.float32, device=A.device)
    _dev(Ct, torch.float32, "Ct", 2)
    _dev(C, torch.float32, "C", 2)
    sp = None
    if status is not None:
        _dev(status, torch.int32, "status")
        sp = status.data_ptr()
    _check(lib().cm_matmat(code.handle, A.data_ptr(), _ld(A, "A"), parity.data_ptr(),
                           _ld(parity, "parity"), Bt.data_ptr(), _ld(Bt, "Bt"), N,
                           Ct.data_ptr(), _ld(Ct, "Ct"), survivors, C.data_ptr(),
                           _ld(C, "C"), sp, _stream()), "cm_matmat")
    return Ct, C


# ---- runtime model (Sec. III-B, III-C, III-D) ----------------------------------

SCHEMES = {"uncoded": 0, "repetition": 1, "mds": 2}


def runtime_mean(scheme: str, n: int, k: int, shift: float = 1.0, rate: float = 1.0) -> float:
    """Expected overall runtime (exact harmonic form) of an uncoded,
    n/k-repetition or (n,k)-MDS coded job under the shifted exponential."""
    out = ctypes.c_double(0.0)
    _check(lib().cm_runtime_mean(SCHEMES[scheme], n, k, shift, rate, ctypes.byref(out)),
           "cm_runtime_mean")
    return float(out.value)


def runtime_cdf(scheme: str, n: int, k: int, t, shift: float = 1.0, rate: float = 1.0):
    """P(T_overall <= t) at the points t."""
    t = np.ascontiguousarray(np.asarray(t, dtype=np.float64).ravel())
    F = np.empty_like(t)
    _check(lib().cm_runtime_cdf(SCHEMES[scheme], n, k, shift, rate,
                                t.ctypes.data_as(ctypes.c_void_p), t.size,
                                F.ctypes.data_as(ctypes.c_void_p)), "cm_runtime_cdf")
    return F


def runtime_simulate(scheme: str, n: int, k: int, count: int, seed: int, counter0: int = 0,
                     shift: float = 1.0, rate: float = 1.0):
    """Monte-Carlo overall runtimes from the straggler draws of draw_erasures."""
    T = np.empty(count, np.float64)
    _check(lib().cm_runtime_simulate(SCHEMES[scheme], n, k, shift, rate, seed, counter0, count,
                                     T.ctypes.data_as(ctypes.c_void_p)), "cm_runtime_simulate")
    return T


def optimal_mds_k(n: int, rate: float = 1.0):
    """(k*, gamma*) of the lemma on optimal MDS-coded algorithms (Lambert W)."""
    ks, g = ctypes.c_double(0.0), ctypes.c_double(0.0)
    _check(lib().cm_optimal_mds_k(n, rate, ctypes.byref(ks), ctypes.byref(g)),
           "cm_optimal_mds_k")
    return float(ks.value), float(g.value)


# ---- coded shuffling (Sec. IV) --------------------------------------------------

SHUFFLE_OPS = {"add": 0, "xor": 1}


class _ShuffleStats(ctypes.Structure):
    _fields_ = [("iteration", ctypes.c_int64), ("message_sets", ctypes.c_int64),
                ("coded_rows", ctypes.c_int64), ("uncoded_rows", ctypes.c_int64),
                ("subtractions", ctypes.c_int64)]


def _rows(t: torch.Tensor, name: str) -> int:
    """Pointer of a CUDA matrix of 4-byte words (fp32 or int32), row-major."""
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError("%s must be a CUDA tensor" % name)
    if t.dtype not in (torch.float32, torch.int32):
        raise TypeError("%s must hold 4-byte words (float32 or int32)" % name)
    _ld(t, name)
    return t.data_ptr()


def _np(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def shuffle_rates(n: int, q: float, s: float):
    """(R_c, R_u) of the coded shuffling rate theorem and eq. for R_u."""
    c, u = ctypes.c_double(0.0), ctypes.c_double(0.0)
    _check(lib().cm_shuffle_rates(n, q, s, ctypes.byref(c), ctypes.byref(u)),
           "cm_shuffle_rates")
    return float(c.value), float(u.value)


class Shuffle:
    """Coded shuffling of q rows over n workers with caches of s rows.

    The planner is host state in libcm; the device workspace for its row
    programs is a torch byte tensor owned by this object."""

    def __init__(self, n: int, q: int, s: int, partition_seed: int, cache_seed: int):
        out = ctypes.c_void_p()
        _check(lib().cm_shuffle_create(n, q, s, partition_seed, cache_seed, ctypes.byref(out)),
               "cm_shuffle_create")
        self._h = out
        self.n, self.q, self.s = n, q, s
        self._ws = None

    def __del__(self):
        h = getattr(self, "_h", None)
        if h and _lib is not None:
            _lib.cm_shuffle_destroy(h)
            self._h = None

    def next(self) -> dict:
        """Plans the next transition; returns its statistics."""
        st = _ShuffleStats()
        _check(lib().cm_shuffle_next(self._h, ctypes.byref(st)), "cm_shuffle_next")
        return {f: int(getattr(st, f)) for f, _ in _ShuffleStats._fields_}

    def stats(self) -> dict:
        st = _ShuffleStats()
        _check(lib().cm_shuffle_query(self._h, ctypes.byref(st)), "cm_shuffle_query")
        return {f: int(getattr(st, f)) for f, _ in _ShuffleStats._fields_}

    def plan(self):
        """(msg_ptr, msg_src, msg_worker, msg_set) of the last transition."""
        st = self.stats()
        ptr = np.empty(st["coded_rows"] + 1, np.int32)
        src = np.empty(st["uncoded_rows"], np.int32)
        wk = np.empty(st["uncoded_rows"], np.int32)
        sets = np.empty(st["coded_rows"], np.uint64)
        _check(lib().cm_shuffle_plan(self._h, _np(ptr), _np(src), _np(wk), _np(sets)),
               "cm_shuffle_plan")
        return ptr, src, wk, sets

    def received(self):
        """(recv_ptr, recv_row): the layout of the received rows Rx."""
        st = self.stats()
        ptr = np.empty(self.n + 1, np.int32)
        rows = np.empty(st["uncoded_rows"], np.int32)
        _check(lib().cm_shuffle_received(self._h, _np(ptr), _np(rows)), "cm_shuffle_received")
        return ptr, rows

    def caches(self):
        """(owner, slot_row): the current partition and cache slot tables."""
        owner = np.empty(self.q, np.int32)
        slots = np.empty(self.n * self.s, np.int32)
        _check(lib().cm_shuffle_caches(self._h, _np(owner), _np(slots)), "cm_shuffle_caches")
        return owner, slots.reshape(self.n, self.s)

    def workspace_bytes(self) -> int:
        return int(lib().cm_shuffle_workspace_bytes(self._h))

    def upload(self, device=None):
        """Copies the current row programs to the device workspace."""
        nb = self.workspace_bytes()
        if self._ws is None:
            self._ws = torch.empty(nb, dtype=torch.uint8,
                                   device=device or torch.device("cuda"))
        _check(lib().cm_shuffle_upload(self._h, ctypes.c_void_p(self._ws.data_ptr()), nb,
                                       _stream()), "cm_shuffle_upload")

    def _wsp(self):
        return ctypes.c_void_p(self._ws.data_ptr() if self._ws is not None else 0)

    # ---- the planner on the device ----

    def device_workspace_bytes(self) -> int:
        return int(lib().cm_shuffle_device_workspace_bytes(self._h))

    def device_init(self, device=None):
        """Moves the state to a device workspace; later transitions are planned
        on the GPU (device_next) and the data plane uses that workspace."""
        nb = self.device_workspace_bytes()
        if nb == 0:
            raise ValueError("the device planner handles n <= 16")
        ws = torch.empty(nb, dtype=torch.uint8, device=device or torch.device("cuda"))
        _check(lib().cm_shuffle_device_init(self._h, ctypes.c_void_p(ws.data_ptr()), nb,
                                            _stream()), "cm_shuffle_device_init")
        self._ws = ws

    def device_next(self) -> dict:
        """Plans the next transition on the device; returns its statistics."""
        st = _ShuffleStats()
        _check(lib().cm_shuffle_device_next(self._h, self._wsp(), self._ws.numel(),
                                            ctypes.byref(st), _stream()),
               "cm_shuffle_device_next")
        return {f: int(getattr(st, f)) for f, _ in _ShuffleStats._fields_}

    def fill(self, A: torch.Tensor, caches: torch.Tensor | None = None) -> torch.Tensor:
        r = A.shape[1]
        if caches is None:
            caches = torch.empty((self.n * self.s, r), dtype=A.dtype, device=A.device)
        _check(lib().cm_shuffle_fill(self._h, self._wsp(), _rows(A, "A"), _ld(A, "A"), r,
                                     _rows(caches, "caches"), _ld(caches, "caches"), _stream()),
               "cm_shuffle_fill")
        return caches

    def encode(self, op: str, A: torch.Tensor, M: torch.Tensor | None = None) -> torch.Tensor:
        r = A.shape[1]
        if M is None:
            M = torch.empty((max(1, self.stats()["coded_rows"]), r), dtype=A.dtype,
                            device=A.device)
        _check(lib().cm_shuffle_encode(self._h, self._wsp(), SHUFFLE_OPS[op], _rows(A, "A"),
                                       _ld(A, "A"), r, _rows(M, "M"), _ld(M, "M"), _stream()),
               "cm_shuffle_encode")
        return M

    def decode(self, op: str, M: torch.Tensor, caches: torch.Tensor, r: int,
               Rx: torch.Tensor | None = None) -> torch.Tensor:
        if Rx is None:
            Rx = torch.empty((max(1, self.stats()["uncoded_rows"]), r), dtype=M.dtype,
                             device=M.device)
        _check(lib().cm_shuffle_decode(self._h, self._wsp(), SHUFFLE_OPS[op], _rows(M, "M"),
                                       _ld(M, "M"), _rows(caches, "caches"),
                                       _ld(caches, "caches"), r, _rows(Rx, "Rx"), _ld(Rx, "Rx"),
                                       _stream()), "cm_shuffle_decode")
        return Rx

    def commit(self, Rx: torch.Tensor, caches: torch.Tensor, r: int) -> None:
        _check(lib().cm_shuffle_commit(self._h, self._wsp(), _rows(Rx, "Rx"), _ld(Rx, "Rx"), r,
                                       _rows(caches, "caches"), _ld(caches, "caches"),
                                       _stream()), "cm_shuffle_commit")
