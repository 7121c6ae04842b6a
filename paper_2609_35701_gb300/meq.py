"""Thin ctypes binding of the MeqMuon C ABI (include/meq.h).

Argument marshalling only: every step of the optimizer runs in the CUDA
library. There is no fallback: if libmeq.so is missing or fails to load,
importing this module raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmeq.so")

MEQ_OK = 0
STATUS_NAMES = {
    0: "MEQ_OK", 1: "MEQ_ERR_INVALID_ARG", 2: "MEQ_ERR_OOM", 3: "MEQ_ERR_CUDA",
    4: "MEQ_ERR_NONFINITE", 5: "MEQ_ERR_TIMEOUT", 6: "MEQ_ERR_UNSUPPORTED", 7: "MEQ_ERR_CORRUPTED",
}
ROW, COL = 0, 1


class MeqShape(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int64), ("cols", ctypes.c_int64)]


class MeqOptions(ctypes.Structure):
    _fields_ = [
        ("rho", ctypes.c_float),
        ("ns_steps", ctypes.c_int),
        ("ns_a", ctypes.c_float),
        ("ns_b", ctypes.c_float),
        ("ns_c", ctypes.c_float),
        ("nesterov", ctypes.c_int),
        ("ns_fp16_mask", ctypes.c_uint32),
        ("tie_atol", ctypes.c_float),
        ("use_graph", ctypes.c_int),
        ("workspace_limit_bytes", ctypes.c_int64),
        ("wait_timeout_ms", ctypes.c_float),
        ("ns_cta_pair", ctypes.c_int),
        ("ns_x0_fused", ctypes.c_int),
        ("update_rule", ctypes.c_int),
        ("debug_canaries", ctypes.c_int),
        ("debug_skip_load", ctypes.c_int),
    ]


EXPORTED = [
    "meq_default_options", "meq_state_bytes", "meq_init_state", "meq_step", "meq_sync", "meq_free",
    "meq_last_error", "meq_status_string", "meq_read_momentum", "meq_write_momentum",
    "meq_read_ns_output", "meq_read_stats", "meq_kernels_per_step", "meq_debug_wait_selftest",
    "meq_set_profiling", "meq_read_profile", "meq_row_col_stats_noalloc",
    "meq_init_state_kinds", "meq_state_bytes_kinds", "meq_ns_gemm_launches_per_step",
    "meq_read_direction_counts", "meq_reset_direction_counts", "meq_ns_cv_trajectory",
    "meq_check_canaries", "meq_canary_count", "meq_debug_corrupt_canary",
    "meq_step_prepare", "meq_step_apply", "meq_read_update",
]
HIDDEN, REMAINING_2D, VECTOR = 0, 1, 2  # meq_kind
RULE_MEQMUON, RULE_MUON = 0, 1          # meq_update_rule


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with paper_2609_35701_gb300.build.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P, I, F, D = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_double
    lib.meq_default_options.argtypes = [ctypes.POINTER(MeqOptions)]
    lib.meq_default_options.restype = None
    lib.meq_state_bytes.argtypes = [ctypes.POINTER(MeqShape), I, ctypes.POINTER(MeqOptions),
                                    ctypes.POINTER(ctypes.c_size_t), ctypes.POINTER(ctypes.c_size_t)]
    lib.meq_state_bytes.restype = I
    lib.meq_init_state.argtypes = [ctypes.POINTER(MeqShape), I, ctypes.POINTER(MeqOptions), P, ctypes.POINTER(P)]
    lib.meq_init_state.restype = I
    lib.meq_step.argtypes = [ctypes.POINTER(P), ctypes.POINTER(P), P, ctypes.POINTER(MeqShape), I, F, F, F, F, P]
    lib.meq_step.restype = I
    lib.meq_step_prepare.argtypes = [ctypes.POINTER(P), P, ctypes.POINTER(MeqShape), I, F, F, F, F, P]
    lib.meq_step_prepare.restype = I
    lib.meq_step_apply.argtypes = [ctypes.POINTER(P), P, P]
    lib.meq_step_apply.restype = I
    lib.meq_sync.argtypes = [P]
    lib.meq_sync.restype = I
    lib.meq_free.argtypes = [P]
    lib.meq_free.restype = I
    lib.meq_last_error.argtypes = [P]
    lib.meq_last_error.restype = ctypes.c_char_p
    lib.meq_status_string.argtypes = [I]
    lib.meq_status_string.restype = ctypes.c_char_p
    lib.meq_read_momentum.argtypes = [P, I, P]
    lib.meq_read_momentum.restype = I
    lib.meq_write_momentum.argtypes = [P, I, P]
    lib.meq_write_momentum.restype = I
    lib.meq_read_ns_output.argtypes = [P, I, P]
    lib.meq_read_ns_output.restype = I
    lib.meq_read_update.argtypes = [P, I, P]
    lib.meq_read_update.restype = I
    lib.meq_read_stats.argtypes = [P, I, P, P, ctypes.POINTER(D), ctypes.POINTER(D), ctypes.POINTER(I)]
    lib.meq_read_stats.restype = I
    lib.meq_kernels_per_step.argtypes = [P]
    lib.meq_kernels_per_step.restype = I
    lib.meq_debug_wait_selftest.argtypes = [P, F]
    lib.meq_debug_wait_selftest.restype = I
    lib.meq_set_profiling.argtypes = [P, I]
    lib.meq_set_profiling.restype = I
    lib.meq_read_profile.argtypes = [P, P, ctypes.POINTER(ctypes.c_int64)]
    lib.meq_read_profile.restype = I
    lib.meq_row_col_stats_noalloc.argtypes = [P, ctypes.c_int64, ctypes.c_int64, F, F, P, P, P, P, P]
    lib.meq_row_col_stats_noalloc.restype = I
    lib.meq_init_state_kinds.argtypes = [ctypes.POINTER(MeqShape), P, I, ctypes.POINTER(MeqOptions), P,
                                         ctypes.POINTER(P)]
    lib.meq_init_state_kinds.restype = I
    lib.meq_state_bytes_kinds.argtypes = [ctypes.POINTER(MeqShape), P, I, ctypes.POINTER(MeqOptions),
                                          ctypes.POINTER(ctypes.c_size_t), ctypes.POINTER(ctypes.c_size_t)]
    lib.meq_state_bytes_kinds.restype = I
    lib.meq_ns_gemm_launches_per_step.argtypes = [P]
    lib.meq_ns_gemm_launches_per_step.restype = I
    lib.meq_read_direction_counts.argtypes = [P, I, ctypes.POINTER(ctypes.c_int64), ctypes.POINTER(ctypes.c_int64)]
    lib.meq_read_direction_counts.restype = I
    lib.meq_reset_direction_counts.argtypes = [P]
    lib.meq_reset_direction_counts.restype = I
    lib.meq_ns_cv_trajectory.argtypes = [P, ctypes.c_int64, ctypes.c_int64, I, F, ctypes.POINTER(MeqOptions),
                                         ctypes.POINTER(D), ctypes.POINTER(D), P]
    lib.meq_ns_cv_trajectory.restype = I
    lib.meq_check_canaries.argtypes = [P, ctypes.POINTER(ctypes.c_int64)]
    lib.meq_check_canaries.restype = I
    lib.meq_canary_count.argtypes = [P]
    lib.meq_canary_count.restype = I
    lib.meq_debug_corrupt_canary.argtypes = [P, I]
    lib.meq_debug_corrupt_canary.restype = I
    return lib


lib = _load()


class MeqError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def default_options(**overrides):
    o = MeqOptions()
    lib.meq_default_options(ctypes.byref(o))
    for k, v in overrides.items():
        if not hasattr(o, k):
            raise KeyError(k)
        setattr(o, k, v)
    return o


def _shape_array(shapes):
    arr = (MeqShape * len(shapes))()
    for i, (r, c) in enumerate(shapes):
        arr[i].rows, arr[i].cols = int(r), int(c)
    return arr


def _kind_array(kinds, n):
    if kinds is None:
        return None
    if len(kinds) != n:
        raise ValueError("one kind per shape")
    return (ctypes.c_int * n)(*[int(k) for k in kinds])


def state_bytes(shapes, kinds=None, **opts):
    """(persistent, workspace) bytes for a shape list, computed on the host."""
    p, w = ctypes.c_size_t(), ctypes.c_size_t()
    o = default_options(**opts)
    st = lib.meq_state_bytes_kinds(_shape_array(shapes), _kind_array(kinds, len(shapes)), len(shapes), ctypes.byref(o),
                                   ctypes.byref(p), ctypes.byref(w))
    if st != MEQ_OK:
        raise MeqError(st, lib.meq_last_error(None).decode())
    return p.value, w.value


def ns_cv_trajectory(H, steps=20, eps=1e-7, stream=None, **opts):
    """(gamma_r, gamma_c) of the NS iterates X_0..X_steps of a CUDA fp32
    matrix H (meq_ns_cv_trajectory)."""
    if H.dim() != 2:
        raise ValueError("H must be a matrix")
    _require_cuda(H, "float32", H.shape[0] * H.shape[1], "H")
    gr = (ctypes.c_double * (steps + 1))()
    gc = (ctypes.c_double * (steps + 1))()
    o = default_options(**opts)
    st = lib.meq_ns_cv_trajectory(H.data_ptr(), H.shape[0], H.shape[1], int(steps), float(eps), ctypes.byref(o),
                                  gr, gc, _stream_handle(stream))
    if st != MEQ_OK:
        raise MeqError(st, lib.meq_last_error(None).decode())
    return np.array(list(gr)), np.array(list(gc))


def row_col_stats_noalloc(U, r, c, gammas, direction, eps=1e-7, tie_atol=1e-6, stream=None):
    """Statistics of one CUDA fp32 matrix U into caller-provided CUDA tensors
    r (rows), c (cols), gammas (2 x float64) and direction (1 x int32),
    without any device allocation (see include/meq.h). Returns the status."""
    rows, cols = U.shape
    _require_cuda(U, "float32", rows * cols, "U")
    _require_cuda(r, "float32", rows, "r", U.device.index)
    _require_cuda(c, "float32", cols, "c", U.device.index)
    _require_cuda(gammas, "float64", 2, "gammas", U.device.index)
    _require_cuda(direction, "int32", 1, "direction", U.device.index)
    return lib.meq_row_col_stats_noalloc(ctypes.c_void_p(U.data_ptr()), rows, cols, float(eps), float(tie_atol),
                                         ctypes.c_void_p(r.data_ptr()), ctypes.c_void_p(c.data_ptr()),
                                         ctypes.c_void_p(gammas.data_ptr()), ctypes.c_void_p(direction.data_ptr()),
                                         _stream_handle(stream))


def _require_cuda(t, dtype_name, numel, what, device=None):
    """Raises unless t is a contiguous CUDA tensor of the given dtype (a
    torch dtype name) and element count (on `device` when given): the library
    only sees a pointer, so a tensor of the wrong size or type would be read
    or written past its end."""
    if not t.is_cuda or str(t.dtype) != "torch." + dtype_name or not t.is_contiguous():
        raise ValueError(f"{what} must be a contiguous {dtype_name} CUDA tensor")
    if t.numel() != numel:
        raise ValueError(f"{what} has {t.numel()} elements, expected {numel}")
    if device is not None and t.device.index != device:
        raise ValueError(f"{what} is on cuda:{t.device.index}, the state on cuda:{device}")


def _stream_handle(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


class MeqMuon:
    """MeqMuon state for a fixed list of parameters (rows, cols); kinds (one
    meq_kind per entry, default all HIDDEN) select the branch of Algorithm 1."""

    def __init__(self, shapes, stream=None, kinds=None, **opts):
        self.shapes = [(int(r), int(c)) for r, c in shapes]
        self.kinds = [HIDDEN] * len(self.shapes) if kinds is None else [int(k) for k in kinds]
        self._shape_arr = _shape_array(self.shapes)
        self._opts = default_options(**opts)
        import torch

        self._device = torch.cuda.current_device()  # the state lives on the current device
        self._st = ctypes.c_void_p()
        s = lib.meq_init_state_kinds(self._shape_arr, _kind_array(self.kinds, len(self.shapes)), len(self.shapes),
                                     ctypes.byref(self._opts), _stream_handle(stream), ctypes.byref(self._st))
        if s != MEQ_OK:
            raise MeqError(s, lib.meq_last_error(None).decode())
        n = len(self.shapes)
        self._pp = (ctypes.c_void_p * n)()
        self._gp = (ctypes.c_void_p * n)()

    def _check(self, s):
        if s != MEQ_OK:
            raise MeqError(s, lib.meq_last_error(self._st).decode())

    @property
    def kernels_per_step(self):
        return lib.meq_kernels_per_step(self._st)

    @property
    def ns_gemm_launches_per_step(self):
        return lib.meq_ns_gemm_launches_per_step(self._st)

    def step_ptrs(self, param_ptrs, grad_ptrs, lr, momentum, weight_decay, eps=1e-7, stream=None):
        """One step given raw device pointers (ints)."""
        for i, (p, g) in enumerate(zip(param_ptrs, grad_ptrs)):
            self._pp[i] = p
            self._gp[i] = g
        self._check(lib.meq_step(self._pp, self._gp, self._st, self._shape_arr, len(self.shapes), float(lr),
                                 float(momentum), float(weight_decay), float(eps), _stream_handle(stream)))

    def step(self, params, grads, lr, momentum, weight_decay, eps=1e-7, stream=None):
        """One step on lists of contiguous fp32 CUDA tensors (params updated in place)."""
        if len(params) != len(self.shapes) or len(grads) != len(self.shapes):
            raise ValueError("params / grads must have one tensor per matrix")
        self._check_tensors(params, "params")
        self._check_tensors(grads, "grads")
        self.step_ptrs([p.data_ptr() for p in params], [g.data_ptr() for g in grads], lr, momentum, weight_decay,
                       eps, stream)

    def _check_tensors(self, ts, what):
        for i, (t, (r, c)) in enumerate(zip(ts, self.shapes)):
            _require_cuda(t, "float32", r * c, f"{what}[{i}]", self._device)

    def step_prepare(self, grads, lr, momentum, weight_decay, eps=1e-7, stream=None):
        """First half of a step (meq_step_prepare): momentum, Newton-Schulz and
        statistics for these gradients; the parameters are not touched."""
        if len(grads) != len(self.shapes):
            raise ValueError("grads must have one tensor per matrix")
        self._check_tensors(grads, "grads")
        n = len(self.shapes)
        for i, g in enumerate(grads):
            self._gp[i] = g.data_ptr()
        self._check(lib.meq_step_prepare(self._gp, self._st, self._shape_arr, n, float(lr), float(momentum),
                                         float(weight_decay), float(eps), _stream_handle(stream)))

    def step_apply(self, params, stream=None):
        """Second half of a step (meq_step_apply): the update of params."""
        if len(params) != len(self.shapes):
            raise ValueError("params must have one tensor per matrix")
        self._check_tensors(params, "params")
        for i, p in enumerate(params):
            self._pp[i] = p.data_ptr()
        self._check(lib.meq_step_apply(self._pp, self._st, _stream_handle(stream)))

    def sync(self):
        self._check(lib.meq_sync(self._st))

    def read_momentum(self, i):
        r, c = self.shapes[i]
        out = np.empty((r, c), np.float32)
        self._check(lib.meq_read_momentum(self._st, i, out.ctypes.data))
        return out

    def write_momentum(self, i, arr):
        r, c = self.shapes[i]
        a = np.ascontiguousarray(arr, dtype=np.float32)
        if a.shape != (r, c):
            raise ValueError(f"momentum {i} must have shape {(r, c)}, got {a.shape}")
        self._check(lib.meq_write_momentum(self._st, i, a.ctypes.data))

    def read_ns_output(self, i):
        r, c = self.shapes[i]
        out = np.empty((r, c), np.float32)
        self._check(lib.meq_read_ns_output(self._st, i, out.ctypes.data))
        return out

    def read_update(self, i):
        """The normalised update U~ the last step applied to entry i (meq_read_update)."""
        r, c = self.shapes[i]
        out = np.empty((r, c), np.float32)
        self._check(lib.meq_read_update(self._st, i, out.ctypes.data))
        return out

    def read_stats(self, i):
        r, c = self.shapes[i]
        rv = np.empty(r, np.float32)
        cv = np.empty(c, np.float32)
        gr, gc, d = ctypes.c_double(), ctypes.c_double(), ctypes.c_int()
        self._check(lib.meq_read_stats(self._st, i, rv.ctypes.data, cv.ctypes.data, ctypes.byref(gr),
                                       ctypes.byref(gc), ctypes.byref(d)))
        return {"r": rv, "c": cv, "gamma_r": gr.value, "gamma_c": gc.value, "direction": d.value}

    def read_direction_counts(self, i):
        """(row choices, column choices) of Eq. (11) for hidden weight i."""
        r, c = ctypes.c_int64(), ctypes.c_int64()
        self._check(lib.meq_read_direction_counts(self._st, i, ctypes.byref(r), ctypes.byref(c)))
        return r.value, c.value

    def check_canaries(self):
        """Raises MeqError (MEQ_ERR_CORRUPTED) if a workspace guard band changed."""
        off = ctypes.c_int64()
        self._check(lib.meq_check_canaries(self._st, ctypes.byref(off)))

    @property
    def canary_count(self):
        return lib.meq_canary_count(self._st)

    def reset_direction_counts(self):
        self._check(lib.meq_reset_direction_counts(self._st))

    def set_profiling(self, enable):
        self._check(lib.meq_set_profiling(self._st, int(bool(enable))))

    PHASES = ("momentum", "cast_x0", "ns_gemm", "stats", "apply")

    def read_profile(self):
        """Summed per-phase milliseconds and the number of profiled steps."""
        ms = (ctypes.c_double * 5)()
        n = ctypes.c_int64()
        self._check(lib.meq_read_profile(self._st, ms, ctypes.byref(n)))
        return dict(zip(self.PHASES, list(ms))), n.value

    def wait_selftest(self, timeout_ms=200.0):
        """Returns the status of the bounded-wait self test (expected MEQ_ERR_TIMEOUT)."""
        return lib.meq_debug_wait_selftest(self._st, float(timeout_ms))

    def close(self):
        if self._st:
            lib.meq_free(self._st)
            self._st = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
