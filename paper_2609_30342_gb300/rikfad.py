"""Python binding of the R-iKFAD C ABI (``include/rikfad.h``).

Argument marshalling only: every step of the optimiser runs in the CUDA
kernels of ``librikfad.so``.  PyTorch supplies device memory and streams; the
binding passes raw device pointers and the ``cudaStream_t`` of the current
torch stream.  If the library has not been built the binding raises: there
is no fallback implementation.
"""
import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
# RIKFAD_LIBRARY may name another build of the same library (the checked
# build, librikfad_checked.so); it is read when the library is first loaded.
LIB_PATH = os.environ.get("RIKFAD_LIBRARY") or os.path.join(_PKG, "librikfad.so")

OK = 0
ERR_ARG = -1
ERR_ALIGN = -2
ERR_CUDA = -3
ERR_OOM = -4
ERR_NONFINITE = -5
ERR_STATE = -6
GRAD_F32 = 0
GRAD_BF16 = 1


class RikfadError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__("rikfad error %d: %s" % (code, msg))
        self.code = code


class Shape(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int64), ("cols", ctypes.c_int64)]


class HParams(ctypes.Structure):
    _fields_ = [("alpha", ctypes.c_double), ("mu", ctypes.c_double), ("gamma", ctypes.c_double),
                ("eps_stab", ctypes.c_double)]


_lib = None

# (name, restype, argtypes) of every exported symbol of include/rikfad.h
_VP = ctypes.c_void_p
_PP = ctypes.POINTER(ctypes.c_void_p)
SIGNATURES = [
    ("rikfad_create", ctypes.c_int, [ctypes.POINTER(Shape), ctypes.c_int, ctypes.POINTER(HParams),
                                     ctypes.c_int, ctypes.POINTER(_VP)]),
    ("rikfad_create_ikfad", ctypes.c_int, [ctypes.POINTER(Shape), ctypes.c_int,
                                           ctypes.POINTER(HParams), ctypes.c_int,
                                           ctypes.POINTER(_VP)]),
    ("rikfad_create_ikfad_shadow", ctypes.c_int, [ctypes.POINTER(Shape), ctypes.c_int,
                                                  ctypes.POINTER(HParams), ctypes.c_int,
                                                  ctypes.POINTER(_VP)]),
    ("rikfad_destroy", None, [_VP]),
    ("rikfad_step", ctypes.c_int, [_VP, ctypes.c_double, _PP, _PP, _PP, _VP]),
    ("rikfad_materialize", ctypes.c_int, [_VP, _PP, _VP]),
    ("rikfad_canonical_momentum", ctypes.c_int, [_VP, _PP, _PP, _VP]),
    ("rikfad_state_bytes", ctypes.c_size_t, [_VP, ctypes.c_int]),
    ("rikfad_state_bytes_for", ctypes.c_size_t, [ctypes.POINTER(Shape), ctypes.c_int, ctypes.c_int]),
    ("rikfad_workspace_bytes", ctypes.c_size_t, [_VP]),
    ("rikfad_pending_step", ctypes.c_double, [_VP]),
    ("rikfad_get_factors", ctypes.c_int, [_VP, ctypes.c_int, _VP, _VP]),
    ("rikfad_set_factors", ctypes.c_int, [_VP, ctypes.c_int, _VP, _VP]),
    ("rikfad_read_denominators", ctypes.c_int, [_VP, _VP, _VP]),
    ("rikfad_enqueue_denominators", ctypes.c_int, [_VP, _VP, _VP]),
    ("rikfad_get_friction", ctypes.c_int, [_VP, ctypes.c_int, _VP]),
    ("rikfad_friction_diagnostics", ctypes.c_int, [_VP, ctypes.c_int, ctypes.c_int, ctypes.c_double,
                                                   ctypes.POINTER(ctypes.c_double), _VP]),
    ("rikfad_state_image_bytes", ctypes.c_size_t, [_VP]),
    ("rikfad_export_state", ctypes.c_int, [_VP, _VP, _VP]),
    ("rikfad_import_state", ctypes.c_int, [_VP, _VP, _VP]),
    ("rikfad_profile_enable", ctypes.c_int, [_VP, ctypes.c_int]),
    ("rikfad_profile_read", ctypes.c_int, [_VP, ctypes.POINTER(ctypes.c_double),
                                           ctypes.POINTER(ctypes.c_double),
                                           ctypes.POINTER(ctypes.c_int64)]),
    ("rikfad_launches_per_step", ctypes.c_int, [_VP]),
    ("rikfad_check_finite", ctypes.c_int, [_VP, _VP]),
    ("rikfad_debug_check_failures", ctypes.c_int, [_VP, ctypes.POINTER(ctypes.c_int64),
                                                   ctypes.POINTER(ctypes.c_int)]),
    ("rikfad_debug_fail_allocation", None, [ctypes.c_int64]),
    ("rikfad_debug_live_allocations", ctypes.c_int64, []),
    ("rikfad_plan_query", ctypes.c_int64, [ctypes.POINTER(Shape), ctypes.c_int, ctypes.c_int,
                                           ctypes.c_int, ctypes.POINTER(ctypes.c_int64),
                                           ctypes.c_int64]),
    ("rikfad_step_matrix_noalloc", ctypes.c_int, [ctypes.c_int64, ctypes.c_int64, ctypes.c_double,
                                                  ctypes.c_double, ctypes.POINTER(HParams),
                                                  ctypes.c_int, _VP, _VP, _VP, _VP, _VP, _VP]),
    ("rikfad_quadratic_run", ctypes.c_int, [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, _VP, _VP,
                                            _VP, _VP, _VP, ctypes.c_double, ctypes.POINTER(HParams),
                                            ctypes.c_int64, _VP, ctypes.c_int64, _VP, _VP]),
    ("rikfad_last_error", ctypes.c_char_p, []),
    ("rikfad_abi_version", ctypes.c_int, []),
]


def lib():
    """Load librikfad.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("%s is missing: build it with paper_2609_30342_gb300.build.build()"
                               % LIB_PATH)
        L = ctypes.CDLL(LIB_PATH)
        for name, res, args in SIGNATURES:
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(rc):
    if rc != OK:
        raise RikfadError(rc, lib().rikfad_last_error().decode(errors="replace"))
    return rc


def _shapes(shapes):
    arr = (Shape * max(len(shapes), 1))()
    for i, (m, n) in enumerate(shapes):
        arr[i].rows = int(m)
        arr[i].cols = int(n)
    return arr


def _stream_ptr(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _ptr_array(tensors):
    return (ctypes.c_void_p * max(len(tensors), 1))(*[_ptr(t) for t in tensors])


def state_bytes_for(shapes, include_momentum=True):
    """Auxiliary state bytes of a shape list (paper's memory-table count)."""
    return lib().rikfad_state_bytes_for(_shapes(shapes), len(shapes), 1 if include_momentum else 0)


def plan_query(shapes, grad_dtype, nblocks):
    """The host planner's pieces: int64 array with rows
    (block, tensor, kind, col0, width, begin, end, slot)."""
    sh = _shapes(shapes)
    gd = GRAD_BF16 if grad_dtype in ("bf16", GRAD_BF16) else GRAD_F32
    n = lib().rikfad_plan_query(sh, len(shapes), gd, int(nblocks), None, 0)
    if n < 0:
        _check(int(n))
    out = np.zeros((max(n, 1), 8), np.int64)
    n2 = lib().rikfad_plan_query(sh, len(shapes), gd, int(nblocks),
                                 out.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), n)
    if n2 != n:
        raise RuntimeError("plan size changed between calls")
    return out[:n]


def _check_tensor(name, t, numel, dtype):
    """Raise ValueError unless ``t`` is a contiguous CUDA tensor of ``dtype``
    with ``numel`` elements (the C side cannot check sizes)."""
    import torch
    if not isinstance(t, torch.Tensor):
        raise ValueError("%s must be a torch tensor" % name)
    if not t.is_cuda:
        raise ValueError("%s must be a CUDA tensor" % name)
    if t.dtype != dtype:
        raise ValueError("%s must be %s, not %s" % (name, dtype, t.dtype))
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if t.numel() != numel:
        raise ValueError("%s has %d elements, expected %d" % (name, t.numel(), numel))


def step_matrix_noalloc(rows, cols, h, pending_step, alpha, mu, gamma, eps_stab, grad_dtype, x, grad,
                        p, R, C, stream=None):
    """One allocation-free step of a single matrix (``rikfad_step_matrix_noalloc``):
    the caller owns x, grad, p and the factors R, C, and remembers the
    previous step size itself (``pending_step``).  Sizes within the library's
    limits are checked here: x, p (float32) and grad (bf16 or float32, as
    ``grad_dtype``) must hold rows * cols elements, R rows and C cols float32
    elements, all contiguous CUDA tensors.  Sizes beyond the limits are left
    to the library, which refuses them."""
    import torch
    hp = HParams(float(alpha), float(mu), float(gamma), float(eps_stab))
    gd = GRAD_BF16 if grad_dtype in ("bf16", GRAD_BF16) else GRAD_F32
    rows, cols = int(rows), int(cols)
    if 0 <= rows <= 65536 and 1 <= cols <= 1024:
        gdt = torch.bfloat16 if gd == GRAD_BF16 else torch.float32
        for name, t, n, dt in (("x", x, rows * cols, torch.float32), ("p", p, rows * cols, torch.float32),
                               ("grad", grad, rows * cols, gdt), ("R", R, rows, torch.float32),
                               ("C", C, cols, torch.float32)):
            _check_tensor(name, t, n, dt)
    _check(lib().rikfad_step_matrix_noalloc(int(rows), int(cols), float(h), float(pending_step),
                                            ctypes.byref(hp), gd, _ptr(x), _ptr(grad), _ptr(p),
                                            _ptr(R), _ptr(C), _stream_ptr(stream)))


def quadratic_run(A, X, P, R, C, h, alpha, mu, gamma, eps_stab, nsteps, record=None, energy=None,
                  stream=None):
    """Batched BACD integration on dense quadratics (``rikfad_quadratic_run``).

    ``A`` is (batch, m n, m n), ``X`` and ``P`` (batch, m, n), ``R`` (batch, m),
    ``C`` (batch, n): contiguous float32 CUDA tensors; X, P, R, C are advanced
    in place.  ``record`` is an int64 CUDA tensor of ascending step indices and
    ``energy`` a (len(record), batch) float32 CUDA tensor that receives the
    energies."""
    batch, m, n = X.shape
    for t in (A, X, P, R, C) + ((record, energy) if record is not None else ()):
        if not t.is_contiguous():
            raise ValueError("quadratic_run needs contiguous tensors")
    if tuple(A.shape) != (batch, m * n, m * n) or tuple(P.shape) != (batch, m, n) \
            or tuple(R.shape) != (batch, m) or tuple(C.shape) != (batch, n):
        raise ValueError("quadratic_run: inconsistent shapes")
    nrec = 0
    if record is not None:
        nrec = record.numel()
        if energy is None or tuple(energy.shape) != (nrec, batch):
            raise ValueError("energy must be (len(record), batch)")
    hp = HParams(float(alpha), float(mu), float(gamma), float(eps_stab))
    _check(lib().rikfad_quadratic_run(int(batch), int(m), int(n), _ptr(A), _ptr(X), _ptr(P), _ptr(R),
                                      _ptr(C), float(h), ctypes.byref(hp), int(nsteps), _ptr(record),
                                      int(nrec), _ptr(energy), _stream_ptr(stream)))


def pointer_array(tensors):
    """A packed host array of the tensors' device pointers (kept alive by the
    caller together with the tensors)."""
    return _ptr_array(tensors)


class PointerSet:
    """Pointer arrays for one (x, grad, p) tensor set, packed once."""

    def __init__(self, x, grad, p):
        self.keep = (list(x), list(grad), list(p))
        self.x = _ptr_array(x)
        self.g = _ptr_array(grad)
        self.p = _ptr_array(p)


class RIKFAD:
    """An R-iKFAD optimiser over a fixed list of parameter tensors.

    ``shapes``: list of ``(rows, cols)``; ``cols == 0`` marks a tensor that is
    not a matrix (``rows`` elements, element-wise rule).  Hyperparameters as
    in the paper (Section 2): ``alpha`` factor decay, ``mu`` friction scale,
    ``gamma`` linear damping, ``eps_stab`` stabiliser.  ``method="ikfad"``
    creates full-friction iKFAD instead (element-wise friction on every
    tensor, ``rikfad_create_ikfad``); ``method="ikfad_shadow"`` runs full
    iKFAD with R-iKFAD's factors carried as shadows (``rikfad_create_ikfad_shadow``,
    for ``friction_diagnostics``).
    """

    def __init__(self, shapes, alpha, mu, gamma=0.0, eps_stab=1e-16, grad_dtype="bf16",
                 method="rikfad"):
        if method not in ("rikfad", "ikfad", "ikfad_shadow"):
            raise ValueError("method must be 'rikfad', 'ikfad' or 'ikfad_shadow'")
        self.method = method
        self.shapes = [(int(m), int(n)) for m, n in shapes]
        self.grad_dtype = GRAD_BF16 if grad_dtype in ("bf16", GRAD_BF16) else GRAD_F32
        hp = HParams(float(alpha), float(mu), float(gamma), float(eps_stab))
        h = ctypes.c_void_p()
        create = {"rikfad": lib().rikfad_create, "ikfad": lib().rikfad_create_ikfad,
                  "ikfad_shadow": lib().rikfad_create_ikfad_shadow}[method]
        _check(create(_shapes(self.shapes), len(self.shapes), ctypes.byref(hp), self.grad_dtype,
                      ctypes.byref(h)))
        self._h = h

    @property
    def handle(self):
        if self._h is None:
            raise RuntimeError("optimiser is closed")
        return self._h

    def close(self):
        if getattr(self, "_h", None) is not None:
            lib().rikfad_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def pack(self, x, grad, p):
        if not (len(x) == len(grad) == len(p) == len(self.shapes)):
            raise ValueError("need one x, grad and p per tensor")
        return PointerSet(x, grad, p)

    def step(self, h, x=None, grad=None, p=None, stream=None, ptrs=None):
        """Enqueue one step of size ``h`` (x, grad, p: lists of CUDA tensors,
        or a ``PointerSet`` from ``pack``)."""
        if ptrs is None:
            ptrs = self.pack(x, grad, p)
        _check(lib().rikfad_step(self.handle, float(h), ptrs.x, ptrs.g, ptrs.p,
                                 _stream_ptr(stream)))

    def materialize(self, p, stream=None):
        """Make the stored momenta canonical in place (``rikfad_materialize``);
        ``p`` is a list of tensors or an array from ``pointer_array``."""
        arr = p if isinstance(p, ctypes.Array) else _ptr_array(p)
        _check(lib().rikfad_materialize(self.handle, arr, _stream_ptr(stream)))

    def canonical_momentum(self, p, out, stream=None):
        _check(lib().rikfad_canonical_momentum(self.handle, _ptr_array(p), _ptr_array(out),
                                               _stream_ptr(stream)))

    def state_bytes(self, include_momentum=True):
        return lib().rikfad_state_bytes(self.handle, 1 if include_momentum else 0)

    def workspace_bytes(self):
        return lib().rikfad_workspace_bytes(self.handle)

    @property
    def pending_step(self):
        return lib().rikfad_pending_step(self.handle)

    def get_factors(self, t):
        """(R, C) of matrix t, or (friction, None) of a vector (of every tensor,
        flattened, under full-friction iKFAD), as float32 numpy."""
        if not 0 <= t < len(self.shapes):
            raise RikfadError(ERR_ARG, "tensor index %d out of range" % t)
        m, n = self.shapes[t]
        if self.method == "ikfad":
            m, n = (m if n == 0 else m * n), 0
        R = np.zeros(m, np.float32)
        C = np.zeros(n, np.float32) if n else None
        _check(lib().rikfad_get_factors(self.handle, int(t), R.ctypes.data if m else None,
                                        C.ctypes.data if n else None))
        return R, C

    def set_factors(self, t, R, C=None):
        R = np.ascontiguousarray(R, np.float32)
        Cp = None
        if C is not None:
            C = np.ascontiguousarray(C, np.float32)
            Cp = C.ctypes.data if C.size else None
        _check(lib().rikfad_set_factors(self.handle, int(t), R.ctypes.data if R.size else None, Cp))

    def get_friction(self, t):
        """Element-wise friction of tensor t (vector, or matrix of a shadow
        handle) as float32 numpy of the tensor's shape."""
        if not 0 <= t < len(self.shapes):
            raise RikfadError(ERR_ARG, "tensor index %d out of range" % t)
        m, n = self.shapes[t]
        out = np.zeros(m if n == 0 else (m, n), np.float32)
        _check(lib().rikfad_get_friction(self.handle, int(t), out.ctypes.data if out.size else 0))
        return out

    def friction_diagnostics(self, t, max_iters=200, tol=1e-10, stream=None):
        """(rel_err, eckart_young_floor, stable_rank, sigma1, frob, iterations)
        of matrix t of a shadow handle."""
        out = (ctypes.c_double * 6)()
        _check(lib().rikfad_friction_diagnostics(self.handle, int(t), int(max_iters), float(tol), out,
                                                 _stream_ptr(stream)))
        return tuple(out)

    def read_denominators(self, stream=None):
        out = np.zeros(max(len(self.shapes), 1), np.float32)
        _check(lib().rikfad_read_denominators(self.handle, out.ctypes.data, _stream_ptr(stream)))
        return out[:len(self.shapes)]

    def enqueue_denominators(self, out, stream=None):
        """Enqueue the read-back of the friction denominators into ``out``, a
        page-locked float32 CPU tensor of at least len(shapes) elements;
        the values are there once ``stream`` passes this point."""
        import torch
        if not (isinstance(out, torch.Tensor) and out.device.type == "cpu" and out.is_pinned() and
                out.dtype == torch.float32 and out.is_contiguous() and out.numel() >= len(self.shapes)):
            raise ValueError("out must be a contiguous page-locked float32 CPU tensor of at least %d "
                             "elements" % len(self.shapes))
        _check(lib().rikfad_enqueue_denominators(self.handle, out.data_ptr(), _stream_ptr(stream)))

    def state_image_bytes(self):
        return lib().rikfad_state_image_bytes(self.handle)

    def export_state(self, dst, stream=None):
        _check(lib().rikfad_export_state(self.handle, _ptr(dst), _stream_ptr(stream)))

    def import_state(self, src, stream=None):
        _check(lib().rikfad_import_state(self.handle, _ptr(src), _stream_ptr(stream)))

    def profile_enable(self, enable=True):
        _check(lib().rikfad_profile_enable(self.handle, 1 if enable else 0))

    def profile_read(self):
        """(step-kernel ms, finalise-kernel ms, steps) summed since enable."""
        a, b, n = ctypes.c_double(), ctypes.c_double(), ctypes.c_int64()
        _check(lib().rikfad_profile_read(self.handle, ctypes.byref(a), ctypes.byref(b),
                                         ctypes.byref(n)))
        return a.value, b.value, n.value

    def launches_per_step(self):
        return lib().rikfad_launches_per_step(self.handle)

    def check_finite(self, stream=None):
        """Wait for the stream; raise RikfadError(ERR_NONFINITE) if a step
        produced a non-finite factor, friction or denominator (the report is
        then cleared)."""
        _check(lib().rikfad_check_finite(self.handle, _stream_ptr(stream)))

    def debug_check_failures(self):
        """(failed device checks, code of the first); (-1, 0) in a library
        built without the checks."""
        n, code = ctypes.c_int64(), ctypes.c_int()
        _check(lib().rikfad_debug_check_failures(self.handle, ctypes.byref(n), ctypes.byref(code)))
        return n.value, code.value


def debug_fail_allocation(n):
    """Make the n-th library allocation from now on fail (n <= 0: off)."""
    lib().rikfad_debug_fail_allocation(int(n))


def debug_live_allocations():
    """Allocations the library currently holds."""
    return lib().rikfad_debug_live_allocations()
