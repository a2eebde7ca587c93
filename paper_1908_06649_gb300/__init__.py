"""Python binding of the GB300 batched complex DFT (C ABI in include/tcu_dft.h).

Argument marshalling only: every step of the transform runs in the CUDA
library ``libtcu_dft.so`` built from ``csrc/tcu_dft.cu``.  There is no CPU or
PyTorch fallback: if the library is missing this module raises on import of
the library (``lib()``), and a transform on a machine without the library
fails loudly.

The transform is the paper's (arXiv 1908.06649, Sec. 4.5): y = x^T W,
W[r][c] = exp(-(2 pi i/n) r c), computed as n = r^k radix-r stages, each a
tall-left tensor-core product with F_r (Theorem 7).
"""
from __future__ import annotations

import ctypes
import os

from . import _build

TF32 = 1
X3TF32 = 3
BF16 = 4
X3BF16 = 5
FORWARD = -1
INVERSE = 1

OK = 0
ERR_INVALID = 1
ERR_UNSUPPORTED = 2
ERR_CUDA = 3
ERR_OOM = 4
ERR_TIMEOUT = 5
ERR_TOO_LARGE = 6
ERR_BOUNDS = 7

PLAN_DEFAULT = 0
PLAN_NO_FUSE = 1
PLAN_FUSE = 2
PLAN_ONE_PASS = 4

SYMBOLS = (
    "tcu_dft_plan", "tcu_dft_plan_ex", "tcu_dft_is_fused", "tcu_dft_exec",
    "tcu_dft_exec_dir", "tcu_dft_exec_timed",
    "tcu_dft_exec_host", "tcu_dft_exec_noalloc", "tcu_dft_exec_stalled",
    "tcu_dft_check", "tcu_dft_destroy", "tcu_dft_num_passes",
    "tcu_dft_pass_stages", "tcu_dft_plan_passes", "tcu_dft_last_error",
    "tcu_dft_strerror",
    "tcu_dft2_plan", "tcu_dft2_exec", "tcu_conv2_exec", "tcu_dft2_check",
    "tcu_dft2_destroy", "tcu_stencil_plan", "tcu_stencil_weights",
    "tcu_stencil_exec", "tcu_stencil_check", "tcu_stencil_destroy",
    "tcu_stencil_tiles",
)

_lib = None


class TcuDftError(RuntimeError):
    def __init__(self, status, what):
        self.status = status
        super().__init__("%s: %s (status %d)" % (what, strerror(status), status))


def lib_path() -> str:
    """The library this process uses: libtcu_dft.so, or the bounds-checked
    libtcu_dft_checked.so when TCU_DFT_CHECKED=1 is set before the first
    ``lib()`` call."""
    if os.environ.get("TCU_DFT_CHECKED") == "1":
        return _build.CHECKED_LIB_PATH
    return _build.LIB_PATH


def lib():
    """Load the library (built in-tree by ``_build.build()``)."""
    global _lib
    if _lib is not None:
        return _lib
    path = lib_path()
    if not os.path.exists(path):
        raise ImportError(
            "%s is not built; run paper_1908_06649_gb300._build.build_all() "
            "first" % path)
    L = ctypes.CDLL(path)
    vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
    L.tcu_dft_plan.argtypes = [i64, i64, i32, i32]
    L.tcu_dft_plan.restype = vp
    L.tcu_dft_plan_ex.argtypes = [i64, i64, i32, i32, ctypes.c_uint32]
    L.tcu_dft_plan_ex.restype = vp
    L.tcu_dft_is_fused.argtypes = [vp]
    L.tcu_dft_is_fused.restype = ctypes.c_int
    L.tcu_dft_exec.argtypes = [vp, vp, vp, vp]
    L.tcu_dft_exec.restype = ctypes.c_int
    L.tcu_dft_exec_dir.argtypes = [vp, vp, vp, ctypes.c_int, vp]
    L.tcu_dft_exec_dir.restype = ctypes.c_int
    L.tcu_dft_exec_timed.argtypes = [vp, vp, vp, ctypes.c_int, vp,
                                     ctypes.POINTER(vp)]
    L.tcu_dft_exec_timed.restype = ctypes.c_int
    L.tcu_dft_exec_host.argtypes = [vp, vp, vp, vp, ctypes.c_int, vp]
    L.tcu_dft_exec_host.restype = ctypes.c_int
    L.tcu_dft_exec_noalloc.argtypes = [i64, i64, i32, i32, vp, vp, ctypes.c_int,
                                       vp]
    L.tcu_dft_exec_noalloc.restype = ctypes.c_int
    L.tcu_dft_exec_stalled.argtypes = [vp, vp, vp, vp]
    L.tcu_dft_exec_stalled.restype = ctypes.c_int
    L.tcu_dft_check.argtypes = [vp, vp]
    L.tcu_dft_check.restype = ctypes.c_int
    L.tcu_dft_destroy.argtypes = [vp]
    L.tcu_dft_destroy.restype = ctypes.c_int
    L.tcu_dft_num_passes.argtypes = [vp]
    L.tcu_dft_num_passes.restype = ctypes.c_int
    L.tcu_dft_plan_passes.argtypes = [i64, i32, ctypes.POINTER(ctypes.c_int32)]
    L.tcu_dft_plan_passes.restype = ctypes.c_int
    L.tcu_stencil_tiles.argtypes = [i64, i32, i32, ctypes.POINTER(ctypes.c_int64),
                                    ctypes.POINTER(ctypes.c_int64)]
    L.tcu_stencil_tiles.restype = ctypes.c_int64
    L.tcu_dft_pass_stages.argtypes = [vp, ctypes.c_int]
    L.tcu_dft_pass_stages.restype = ctypes.c_int
    L.tcu_dft_last_error.argtypes = []
    L.tcu_dft_last_error.restype = ctypes.c_int
    L.tcu_dft_strerror.argtypes = [ctypes.c_int]
    L.tcu_dft_strerror.restype = ctypes.c_char_p
    L.tcu_dft2_plan.argtypes = [i64, i64, i64, i32, i32]
    L.tcu_dft2_plan.restype = vp
    L.tcu_dft2_exec.argtypes = [vp, vp, vp, ctypes.c_int, vp]
    L.tcu_dft2_exec.restype = ctypes.c_int
    L.tcu_conv2_exec.argtypes = [vp, vp, vp, vp, vp]
    L.tcu_conv2_exec.restype = ctypes.c_int
    fp = ctypes.POINTER(ctypes.c_float)
    L.tcu_stencil_plan.argtypes = [i64, i32, i32, i32]
    L.tcu_stencil_plan.restype = vp
    L.tcu_stencil_weights.argtypes = [vp, fp, vp, vp]
    L.tcu_stencil_weights.restype = ctypes.c_int
    L.tcu_stencil_exec.argtypes = [vp, fp, vp, vp, vp]
    L.tcu_stencil_exec.restype = ctypes.c_int
    for nm in ("tcu_dft2_check", "tcu_stencil_check"):
        getattr(L, nm).argtypes = [vp, vp]
        getattr(L, nm).restype = ctypes.c_int
    for nm in ("tcu_dft2_destroy", "tcu_stencil_destroy"):
        getattr(L, nm).argtypes = [vp]
        getattr(L, nm).restype = ctypes.c_int
    _lib = L
    return L


def plan_passes(n: int, sqrt_m: int = 16):
    """Stages per HBM pass that a plan for (n, sqrt_m) would use ([] if n is
    not supported); no GPU needed."""
    st = (ctypes.c_int32 * 3)()
    np_ = lib().tcu_dft_plan_passes(int(n), int(sqrt_m), st)
    return [int(st[i]) for i in range(np_)]


def stencil_tiles(side: int, steps: int, sqrt_m: int = 16):
    """(tiles, tile side N, output block side B) that tcu_stencil_plan would
    choose; tiles = 0 if unsupported.  Host only: needs no GPU."""
    N = ctypes.c_int64(0)
    B = ctypes.c_int64(0)
    t = lib().tcu_stencil_tiles(int(side), int(steps), int(sqrt_m), ctypes.byref(N),
                                ctypes.byref(B))
    return int(t), int(N.value), int(B.value)


def strerror(status: int) -> str:
    try:
        return lib().tcu_dft_strerror(int(status)).decode()
    except ImportError:
        return "status %d" % status


def _stream_handle(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def exec_noalloc(x, out, n: int, batch: int, sqrt_m: int = 16,
                 precision: int = X3TF32, direction: int = FORWARD, stream=None):
    """tcu_dft_exec_noalloc: the transform without a plan and without any
    device allocation, for callers that must not allocate (its working
    memory is a fixed array inside the library; see include/tcu_dft.h for
    the size limits).  x, out: contiguous complex64 CUDA tensors of batch*n
    elements.  Returns out."""
    import torch
    for t, nm in ((x, "x"), (out, "out")):
        if (not isinstance(t, torch.Tensor) or t.dtype != torch.complex64
                or not t.is_cuda or not t.is_contiguous()
                or t.numel() != n * batch):
            raise ValueError("%s must be a contiguous complex64 CUDA tensor "
                             "of batch*n elements" % nm)
    rc = lib().tcu_dft_exec_noalloc(int(n), int(batch), int(sqrt_m),
                                    int(precision),
                                    ctypes.c_void_p(x.data_ptr()),
                                    ctypes.c_void_p(out.data_ptr()),
                                    int(direction), _stream_handle(stream))
    if rc != OK:
        raise TcuDftError(rc, "tcu_dft_exec_noalloc")
    return out


class Plan:
    """tcu_dft_plan(n, batch, sqrt_m, precision) and its executions.

    ``forward(x)`` / ``inverse(x)`` take a contiguous complex64 CUDA tensor of
    shape (batch, n) (or batch*n elements) and return the transform in a new
    tensor (or in ``out``).  They run on torch's current stream.
    """

    def __init__(self, n: int, batch: int, sqrt_m: int = 16,
                 precision: int = X3TF32, flags: int = PLAN_DEFAULT):
        L = lib()
        h = L.tcu_dft_plan_ex(int(n), int(batch), int(sqrt_m), int(precision),
                              int(flags))
        if not h:
            raise TcuDftError(L.tcu_dft_last_error(), "tcu_dft_plan")
        self._h = h
        self.n, self.batch, self.sqrt_m, self.precision = (
            int(n), int(batch), int(sqrt_m), int(precision))

    @property
    def handle(self):
        return self._h

    @property
    def fused(self) -> bool:
        return lib().tcu_dft_is_fused(self._h) == 1

    def passes(self):
        L = lib()
        return [L.tcu_dft_pass_stages(self._h, i)
                for i in range(L.tcu_dft_num_passes(self._h))]

    def _check_tensor(self, t, name):
        import torch
        if not isinstance(t, torch.Tensor) or t.dtype != torch.complex64:
            raise TypeError("%s must be a complex64 torch tensor" % name)
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError("%s must be a contiguous CUDA tensor" % name)
        if t.numel() != self.n * self.batch:
            raise ValueError("%s must hold batch*n = %d elements"
                             % (name, self.n * self.batch))

    def exec(self, x, out=None, direction: int = FORWARD, stream=None):
        import torch
        self._check_tensor(x, "x")
        if out is None:
            out = torch.empty_like(x)
        self._check_tensor(out, "out")
        rc = lib().tcu_dft_exec_dir(self._h, ctypes.c_void_p(x.data_ptr()),
                                    ctypes.c_void_p(out.data_ptr()),
                                    int(direction), _stream_handle(stream))
        if rc != OK:
            raise TcuDftError(rc, "tcu_dft_exec_dir")
        return out

    def exec_timed(self, x, out, events, direction: int = FORWARD,
                   stream=None):
        """exec() that records torch.cuda.Event objects ``events`` (one per
        pass plus one) around the pass kernels on the stream."""
        self._check_tensor(x, "x")
        self._check_tensor(out, "out")
        arr = (ctypes.c_void_p * len(events))(
            *[ctypes.c_void_p(e.cuda_event) for e in events])
        rc = lib().tcu_dft_exec_timed(self._h, ctypes.c_void_p(x.data_ptr()),
                                      ctypes.c_void_p(out.data_ptr()),
                                      int(direction), _stream_handle(stream),
                                      arr)
        if rc != OK:
            raise TcuDftError(rc, "tcu_dft_exec_timed")
        return out

    def forward(self, x, out=None, stream=None):
        return self.exec(x, out, FORWARD, stream)

    def inverse(self, x, out=None, stream=None):
        return self.exec(x, out, INVERSE, stream)

    def exec_host(self, h_in, h_out, d_work, direction: int = FORWARD,
                  stream=None):
        """Host in -> device work buffer -> host out, all enqueued on the
        stream (synchronise before reading h_out)."""
        self._check_tensor(d_work, "d_work")
        for t, nm in ((h_in, "h_in"), (h_out, "h_out")):
            if t.is_cuda or t.numel() != self.n * self.batch:
                raise ValueError("%s must be a host tensor of batch*n" % nm)
        rc = lib().tcu_dft_exec_host(
            self._h, ctypes.c_void_p(h_in.data_ptr()),
            ctypes.c_void_p(h_out.data_ptr()),
            ctypes.c_void_p(d_work.data_ptr()), int(direction),
            _stream_handle(stream))
        if rc != OK:
            raise TcuDftError(rc, "tcu_dft_exec_host")

    def check(self, stream=None):
        """Synchronise and raise if a device-side wait timed out."""
        rc = lib().tcu_dft_check(self._h, _stream_handle(stream))
        if rc != OK:
            raise TcuDftError(rc, "tcu_dft_check")

    def destroy(self):
        if getattr(self, "_h", None):
            lib().tcu_dft_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def _check_cuda(t, dtype, numel, what):
    import torch
    if (not isinstance(t, torch.Tensor) or t.dtype != dtype or not t.is_cuda
            or not t.is_contiguous() or t.numel() != numel):
        raise ValueError("%s must be a contiguous %s CUDA tensor of %d elements"
                         % (what, dtype, numel))


class Plan2:
    """2-D DFT / circular 2-D convolution plan (tcu_dft2_*): batch row-major
    n1 x n2 complex64 arrays (Sec. 4.6)."""

    def __init__(self, n1: int, n2: int, batch: int, sqrt_m: int = 16,
                 precision: int = X3TF32):
        L = lib()
        self._h = L.tcu_dft2_plan(int(n1), int(n2), int(batch), int(sqrt_m),
                                  int(precision))
        if not self._h:
            raise TcuDftError(L.tcu_dft_last_error(), "tcu_dft2_plan")
        self.n1, self.n2, self.batch = int(n1), int(n2), int(batch)

    def _n(self):
        return self.n1 * self.n2 * self.batch

    def exec(self, x, out=None, direction: int = FORWARD, stream=None):
        import torch
        _check_cuda(x, torch.complex64, self._n(), "x")
        if out is None:
            out = torch.empty_like(x)
        _check_cuda(out, torch.complex64, self._n(), "out")
        rc = lib().tcu_dft2_exec(self._h, ctypes.c_void_p(x.data_ptr()),
                                 ctypes.c_void_p(out.data_ptr()), int(direction),
                                 _stream_handle(stream))
        if rc != OK:
            raise TcuDftError(rc, "tcu_dft2_exec")
        return out

    def forward(self, x, out=None, stream=None):
        return self.exec(x, out, FORWARD, stream)

    def inverse(self, x, out=None, stream=None):
        return self.exec(x, out, INVERSE, stream)

    def conv(self, x, spectrum, out=None, stream=None):
        """IDFT2(DFT2(x) * spectrum) for every array of x."""
        import torch
        _check_cuda(x, torch.complex64, self._n(), "x")
        _check_cuda(spectrum, torch.complex64, self.n1 * self.n2, "spectrum")
        if out is None:
            out = torch.empty_like(x)
        _check_cuda(out, torch.complex64, self._n(), "out")
        rc = lib().tcu_conv2_exec(self._h, ctypes.c_void_p(x.data_ptr()),
                                  ctypes.c_void_p(spectrum.data_ptr()),
                                  ctypes.c_void_p(out.data_ptr()),
                                  _stream_handle(stream))
        if rc != OK:
            raise TcuDftError(rc, "tcu_conv2_exec")
        return out

    def check(self, stream=None):
        rc = lib().tcu_dft2_check(self._h, _stream_handle(stream))
        if rc != OK:
            raise TcuDftError(rc, "tcu_dft2_check")

    def destroy(self):
        if getattr(self, "_h", None):
            lib().tcu_dft2_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


class StencilPlan:
    """Linear (n, k)-stencil on a side x side fp32 grid (tcu_stencil_*):
    the weight matrix by polynomial powering (Lemma 2) and the stencil by
    batched tile convolutions (Lemma 1)."""

    def __init__(self, side: int, steps: int, sqrt_m: int = 16,
                 precision: int = X3TF32):
        L = lib()
        self._h = L.tcu_stencil_plan(int(side), int(steps), int(sqrt_m),
                                     int(precision))
        if not self._h:
            raise TcuDftError(L.tcu_dft_last_error(), "tcu_stencil_plan")
        self.side, self.steps = int(side), int(steps)

    @staticmethod
    def _w3(w3x3):
        vals = [float(v) for row in w3x3 for v in row]
        if len(vals) != 9:
            raise ValueError("w3x3 must be 3 x 3")
        return (ctypes.c_float * 9)(*vals)

    def weights(self, w3x3, out=None, stream=None):
        import torch
        side = 2 * self.steps + 1
        if out is None:
            out = torch.empty(side * side, dtype=torch.float32, device="cuda")
        _check_cuda(out, torch.float32, side * side, "out")
        rc = lib().tcu_stencil_weights(self._h, self._w3(w3x3),
                                       ctypes.c_void_p(out.data_ptr()),
                                       _stream_handle(stream))
        if rc != OK:
            raise TcuDftError(rc, "tcu_stencil_weights")
        return out.reshape(side, side)

    def apply(self, A, out=None, w3x3=None, stream=None):
        import torch
        n = self.side * self.side
        _check_cuda(A, torch.float32, n, "A")
        if out is None:
            out = torch.empty_like(A)
        _check_cuda(out, torch.float32, n, "out")
        rc = lib().tcu_stencil_exec(self._h, self._w3(w3x3),
                                    ctypes.c_void_p(A.data_ptr()),
                                    ctypes.c_void_p(out.data_ptr()),
                                    _stream_handle(stream))
        if rc != OK:
            raise TcuDftError(rc, "tcu_stencil_exec")
        return out

    def check(self, stream=None):
        rc = lib().tcu_stencil_check(self._h, _stream_handle(stream))
        if rc != OK:
            raise TcuDftError(rc, "tcu_stencil_check")

    def destroy(self):
        if getattr(self, "_h", None):
            lib().tcu_stencil_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass
