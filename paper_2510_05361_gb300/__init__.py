"""GB300-native MT-DAO hot path: Python binding of ``libmtdao.so``.

Thin ctypes marshalling over the C ABI declared in ``include/mtdao.h``; the
functions keep the C names (``mtdao_create``, ``mtdao_step``, ``mtdao_sync``,
``mtdao_destroy``, ...).  Every step of the optimizer runs in the library's
CUDA kernels; this module only converts arguments.  PyTorch is used by
callers for device memory and streams.

The library is loaded on first use; if it has not been built (see
``paper_2510_05361_gb300.build``) that first use raises instead of falling
back to anything else.  ``load()`` forces the load.
"""
from __future__ import annotations

import ctypes
import os

from .build import LIB as _LIB_PATH

MAX_MOM = 4
MAX_REPLICAS = 1024

OK, ERR_INVALID, ERR_OOM, ERR_CUDA, ERR_ALIGN, ERR_STATE = 0, -1, -2, -3, -4, -5
BASE_ADAM, BASE_ADOPT, BASE_SGDM = 0, 1, 2
CLIP_NONE, CLIP_GLOBAL_NORM, CLIP_ELEMENTWISE = 0, 1, 2
F32, BF16 = 0, 1
PHASE_ALG1, PHASE_ALG2_LITERAL = 0, 1

BASES = {"adam": BASE_ADAM, "adopt": BASE_ADOPT, "sgdm": BASE_SGDM}
CLIPS = {"none": CLIP_NONE, "global_norm": CLIP_GLOBAL_NORM, "elementwise": CLIP_ELEMENTWISE}
PHASES = {"alg1": PHASE_ALG1, "alg2_literal": PHASE_ALG2_LITERAL}
DTYPES = {"f32": F32, "bf16": BF16}


class mtdao_config(ctypes.Structure):
    _fields_ = [
        ("base", ctypes.c_int32),
        ("n_mom", ctypes.c_int32),
        ("beta1", ctypes.c_double * MAX_MOM),
        ("omega", ctypes.c_double * MAX_MOM),
        ("beta2", ctypes.c_double),
        ("eps", ctypes.c_double),
        ("bias_correction", ctypes.c_int32),
        ("clip_mode", ctypes.c_int32),
        ("clip_rho", ctypes.c_double),
        ("sync_phase", ctypes.c_int32),
        ("period_x", ctypes.c_int64),
        ("period_u", ctypes.c_int64 * MAX_MOM),
        ("period_v", ctypes.c_int64),
        ("adopt_prev_v", ctypes.c_int32),
    ]


class MTDAOError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__("mtdao error %d: %s" % (code, msg))
        self.code = code


def _load():
    if not os.path.exists(_LIB_PATH):
        raise ImportError("libmtdao.so is not built (%s); run "
                          "`python -m paper_2510_05361_gb300.build`" % _LIB_PATH)
    lib = ctypes.CDLL(_LIB_PATH)
    H = ctypes.c_void_p
    cfgp = ctypes.POINTER(mtdao_config)
    i64p = ctypes.POINTER(ctypes.c_int64)
    sig = {
        "mtdao_version": (ctypes.c_int32, []),
        "mtdao_config_default": (ctypes.c_int, [cfgp, ctypes.c_int32, ctypes.c_int32]),
        "mtdao_config_validate": (ctypes.c_int, [cfgp, ctypes.c_int32]),
        "mtdao_num_states": (ctypes.c_int32, [cfgp]),
        "mtdao_plan_layout": (ctypes.c_int, [i64p, ctypes.c_int32, i64p, i64p]),
        "mtdao_due_mask": (ctypes.c_int, [cfgp, ctypes.c_int64, ctypes.POINTER(ctypes.c_uint32)]),
        "mtdao_half_life": (ctypes.c_int, [ctypes.c_double, ctypes.POINTER(ctypes.c_double)]),
        "mtdao_config_half_life_periods": (ctypes.c_int, [cfgp, ctypes.c_int64]),
        "mtdao_comm_reduction": (ctypes.c_int, [cfgp, ctypes.POINTER(ctypes.c_double)]),
        "mtdao_create": (ctypes.c_int, [cfgp, ctypes.c_int32, i64p, ctypes.c_int32, ctypes.c_void_p,
                                        ctypes.POINTER(H)]),
        "mtdao_destroy": (None, [H]),
        "mtdao_set_stream": (ctypes.c_int, [H, ctypes.c_void_p]),
        "mtdao_set_params": (ctypes.c_int, [H, ctypes.c_void_p]),
        "mtdao_step": (ctypes.c_int, [H, ctypes.c_void_p, ctypes.c_int32, ctypes.c_double,
                                      ctypes.c_uint32]),
        "mtdao_step_host": (ctypes.c_int, [H, ctypes.c_void_p, ctypes.c_int32, ctypes.c_double,
                                           ctypes.c_uint32]),
        "mtdao_run": (ctypes.c_int, [H, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32,
                                     ctypes.POINTER(ctypes.c_double), ctypes.c_int32]),
        "mtdao_sync": (ctypes.c_int, [H, ctypes.c_uint32]),
        "mtdao_sync_due": (ctypes.c_int, [H, ctypes.POINTER(ctypes.c_uint32)]),
        "mtdao_sync_stats": (ctypes.c_int, [H, ctypes.c_uint32, ctypes.c_void_p]),
        "mtdao_track_anchor": (ctypes.c_int, [H, ctypes.c_uint32]),
        "mtdao_pseudo_grad_stats": (ctypes.c_int, [H, ctypes.c_int32, ctypes.c_void_p]),
        "mtdao_grad_sqnorm": (ctypes.c_int, [H, ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p]),
        "mtdao_grad_nonfinite": (ctypes.c_int, [H, ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p]),
        "mtdao_grad_sqnorm_static": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32,
                                                    ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]),
        "mtdao_get_state_ptr": (ctypes.c_int, [H, ctypes.c_int32, ctypes.c_int32,
                                               ctypes.POINTER(ctypes.c_void_p)]),
        "mtdao_copy_state_to_host": (ctypes.c_int, [H, ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p]),
        "mtdao_copy_state_from_host": (ctypes.c_int, [H, ctypes.c_int32, ctypes.c_int32,
                                                      ctypes.c_void_p]),
        "mtdao_layout": (ctypes.c_int, [H, i64p, ctypes.POINTER(ctypes.c_int32),
                                        ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int32),
                                        ctypes.POINTER(i64p)]),
        "mtdao_get_step": (ctypes.c_int64, [H]),
        "mtdao_set_step": (ctypes.c_int, [H, ctypes.c_int64]),
        "mtdao_last_error": (ctypes.c_char_p, [H]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


class _LazyLib:
    """Loads libmtdao.so on first attribute access."""

    _handle = None

    def __getattr__(self, name):
        if _LazyLib._handle is None:
            _LazyLib._handle = _load()
        return getattr(_LazyLib._handle, name)


lib = _LazyLib()
LIB_PATH = _LIB_PATH


def load():
    """Load libmtdao.so now (raises ImportError if it is not built)."""
    return lib.mtdao_version()


def _check(rc, h=None):
    if rc != OK:
        raise MTDAOError(rc, (lib.mtdao_last_error(h) or b"").decode())
    return rc


def make_config(opt: dict) -> mtdao_config:
    """mtdao_config from a plain dictionary (base, n_mom, beta1, omega, ...)."""
    c = mtdao_config()
    n = int(opt["n_mom"])
    c.base = BASES[opt["base"]] if isinstance(opt["base"], str) else int(opt["base"])
    c.n_mom = n
    for j in range(n):
        c.beta1[j] = float(opt["beta1"][j])
        c.omega[j] = float(opt["omega"][j])
        c.period_u[j] = int(opt["period_u"][j])
    c.beta2 = float(opt.get("beta2", 0.999))
    c.eps = float(opt.get("eps", 1e-8))
    c.bias_correction = 1 if opt.get("bias_correction", c.base == BASE_ADAM) else 0
    c.clip_mode = CLIPS[opt.get("clip_mode", "none")]
    c.clip_rho = float(opt.get("clip_rho", 1.0))
    c.sync_phase = PHASES[opt.get("sync_phase", "alg1")]
    c.period_x = int(opt["period_x"])
    c.period_v = int(opt.get("period_v", 0))
    c.adopt_prev_v = 1 if opt.get("adopt_prev_v", False) else 0
    return c


# ---- same-name wrappers of the C ABI (argument marshalling only) ----------

def mtdao_version() -> int:
    return int(lib.mtdao_version())


def mtdao_config_default(base: int, n_mom: int) -> mtdao_config:
    c = mtdao_config()
    _check(lib.mtdao_config_default(ctypes.byref(c), base, n_mom))
    return c


def mtdao_config_validate(cfg: mtdao_config, M: int) -> None:
    _check(lib.mtdao_config_validate(ctypes.byref(cfg), M))


def mtdao_num_states(cfg: mtdao_config) -> int:
    return int(lib.mtdao_num_states(ctypes.byref(cfg)))


def mtdao_plan_layout(numels):
    n = len(numels)
    arr = (ctypes.c_int64 * n)(*[int(k) for k in numels])
    offs = (ctypes.c_int64 * n)()
    npad = ctypes.c_int64()
    _check(lib.mtdao_plan_layout(arr, n, offs, ctypes.byref(npad)))
    return list(offs), int(npad.value)


def mtdao_due_mask(cfg: mtdao_config, step: int) -> int:
    m = ctypes.c_uint32()
    _check(lib.mtdao_due_mask(ctypes.byref(cfg), int(step), ctypes.byref(m)))
    return int(m.value)


def mtdao_half_life(beta: float) -> float:
    tau = ctypes.c_double()
    _check(lib.mtdao_half_life(float(beta), ctypes.byref(tau)))
    return float(tau.value)


def mtdao_config_half_life_periods(cfg: mtdao_config, period_x: int) -> mtdao_config:
    """Sets cfg's periods in place (and returns cfg)."""
    _check(lib.mtdao_config_half_life_periods(ctypes.byref(cfg), int(period_x)))
    return cfg


def mtdao_comm_reduction(cfg: mtdao_config) -> float:
    f = ctypes.c_double()
    _check(lib.mtdao_comm_reduction(ctypes.byref(cfg), ctypes.byref(f)))
    return float(f.value)


def mtdao_create(cfg: mtdao_config, M: int, numels, stream: int = 0):
    n = len(numels)
    arr = (ctypes.c_int64 * n)(*[int(k) for k in numels])
    h = ctypes.c_void_p()
    _check(lib.mtdao_create(ctypes.byref(cfg), M, arr, n, ctypes.c_void_p(stream), ctypes.byref(h)))
    return h


def mtdao_destroy(h) -> None:
    lib.mtdao_destroy(h)


def mtdao_set_stream(h, stream: int) -> None:
    _check(lib.mtdao_set_stream(h, ctypes.c_void_p(stream)), h)


def mtdao_set_params(h, x0_dev_ptr: int) -> None:
    _check(lib.mtdao_set_params(h, ctypes.c_void_p(x0_dev_ptr)), h)


def mtdao_step(h, grads_dev_ptr: int, grad_dtype: int, lr: float, sync_mask: int = 0) -> None:
    _check(lib.mtdao_step(h, ctypes.c_void_p(grads_dev_ptr), grad_dtype, float(lr), sync_mask), h)


def mtdao_run(h, grads_dev_ptr: int, grads_stride_bytes: int, grad_dtype: int, lrs) -> None:
    lrs = [float(v) for v in lrs]
    arr = (ctypes.c_double * len(lrs))(*lrs)
    _check(lib.mtdao_run(h, ctypes.c_void_p(grads_dev_ptr), int(grads_stride_bytes), grad_dtype, arr,
                         len(lrs)), h)


def mtdao_step_host(h, grads_host_ptr: int, grad_dtype: int, lr: float, sync_mask: int = 0) -> None:
    _check(lib.mtdao_step_host(h, ctypes.c_void_p(grads_host_ptr), grad_dtype, float(lr), sync_mask), h)


def mtdao_sync(h, mask: int) -> None:
    _check(lib.mtdao_sync(h, mask), h)


def mtdao_sync_stats(h, mask: int, stats_dev_ptr: int) -> None:
    _check(lib.mtdao_sync_stats(h, mask, ctypes.c_void_p(stats_dev_ptr)), h)


def mtdao_track_anchor(h, state_mask: int) -> None:
    _check(lib.mtdao_track_anchor(h, int(state_mask)), h)


def mtdao_pseudo_grad_stats(h, state: int, out_dev_ptr: int) -> None:
    _check(lib.mtdao_pseudo_grad_stats(h, int(state), ctypes.c_void_p(out_dev_ptr)), h)


def mtdao_sync_due(h) -> int:
    m = ctypes.c_uint32()
    _check(lib.mtdao_sync_due(h, ctypes.byref(m)), h)
    return int(m.value)


def mtdao_grad_sqnorm(h, grads_dev_ptr: int, grad_dtype: int, out_dev_ptr: int) -> None:
    _check(lib.mtdao_grad_sqnorm(h, ctypes.c_void_p(grads_dev_ptr), grad_dtype,
                                 ctypes.c_void_p(out_dev_ptr)), h)


def mtdao_grad_nonfinite(h, grads_dev_ptr: int, grad_dtype: int, out_dev_ptr: int) -> None:
    _check(lib.mtdao_grad_nonfinite(h, ctypes.c_void_p(grads_dev_ptr), grad_dtype,
                                    ctypes.c_void_p(out_dev_ptr)), h)


def mtdao_grad_sqnorm_static(grads_dev_ptr: int, grad_dtype: int, M: int, n_padded: int,
                             out_dev_ptr: int, stream: int = 0) -> None:
    """Allocation-free per-replica sum of squares (no handle needed)."""
    _check(lib.mtdao_grad_sqnorm_static(ctypes.c_void_p(grads_dev_ptr), grad_dtype, M, n_padded,
                                        ctypes.c_void_p(out_dev_ptr), ctypes.c_void_p(stream)))


def mtdao_get_state_ptr(h, state: int, replica: int) -> int:
    p = ctypes.c_void_p()
    _check(lib.mtdao_get_state_ptr(h, state, replica, ctypes.byref(p)), h)
    return int(p.value)


def mtdao_copy_state_to_host(h, state: int, replica: int, host_ptr: int) -> None:
    _check(lib.mtdao_copy_state_to_host(h, state, replica, ctypes.c_void_p(host_ptr)), h)


def mtdao_copy_state_from_host(h, state: int, replica: int, host_ptr: int) -> None:
    _check(lib.mtdao_copy_state_from_host(h, state, replica, ctypes.c_void_p(host_ptr)), h)


def mtdao_layout(h) -> dict:
    npad, nt, M, ns = ctypes.c_int64(), ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    offs = ctypes.POINTER(ctypes.c_int64)()
    _check(lib.mtdao_layout(h, ctypes.byref(npad), ctypes.byref(nt), ctypes.byref(M), ctypes.byref(ns),
                            ctypes.byref(offs)), h)
    return {"n_padded": int(npad.value), "n_tensors": int(nt.value), "M": int(M.value),
            "n_states": int(ns.value), "offsets": [int(offs[i]) for i in range(nt.value)]}


def mtdao_get_step(h) -> int:
    return int(lib.mtdao_get_step(h))


def mtdao_set_step(h, step: int) -> None:
    _check(lib.mtdao_set_step(h, int(step)), h)


def mtdao_last_error(h=None) -> str:
    return (lib.mtdao_last_error(h) or b"").decode()


class MTDAO:
    """Owning wrapper of one handle: M replicas of a flattened tensor list.

    ``opt`` is a plain dictionary (see ``make_config``).  Device buffers are
    passed as torch tensors or raw pointers; the stream is torch's current
    stream at construction unless given.
    """

    def __init__(self, opt: dict, M: int, numels, stream: int | None = None):
        import torch
        if stream is None:
            stream = torch.cuda.current_stream().cuda_stream
        self.cfg = make_config(opt)
        self.M = int(M)
        self.h = mtdao_create(self.cfg, self.M, list(numels), stream)
        lay = mtdao_layout(self.h)
        self.n_padded = lay["n_padded"]
        self.n_states = lay["n_states"]
        self.offsets = lay["offsets"]
        self.numels = [int(k) for k in numels]
        self.n_mom = int(opt["n_mom"])

    def close(self) -> None:
        if getattr(self, "h", None) is not None and self.h.value:
            mtdao_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @staticmethod
    def _ptr(t) -> int:
        return t if isinstance(t, int) else int(t.data_ptr())

    def _check_tensor(self, t, what: str, shape, dtypes, device: str) -> None:
        """Tensors are passed as raw pointers, so their layout must be the
        one the library reads: the given shape, one of the dtypes,
        contiguous, on the given kind of device.  Raw integer pointers
        are passed through unchecked."""
        if isinstance(t, int):
            return
        if tuple(t.shape) != tuple(shape) and not (len(shape) == 1 and t.numel() == shape[0] and t.dim() == 1):
            raise ValueError("%s: expected shape %s, got %s" % (what, tuple(shape), tuple(t.shape)))
        if t.dtype not in dtypes:
            raise ValueError("%s: dtype %s not supported" % (what, t.dtype))
        if not t.is_contiguous():
            raise ValueError("%s must be contiguous" % what)
        if (t.device.type == "cuda") != (device == "cuda"):
            raise ValueError("%s must be in %s memory" % (what, "device" if device == "cuda" else "host"))

    def _grad_dtypes(self):
        import torch
        return (torch.float32, torch.bfloat16)

    @staticmethod
    def _grad_code(grads, dtype):
        """The library's dtype code for a gradient buffer: the tensor's own
        (an explicit dtype must agree with it); for a raw pointer the given
        dtype, else F32."""
        if isinstance(grads, int):
            return F32 if dtype is None else dtype
        import torch
        code = BF16 if grads.dtype == torch.bfloat16 else F32
        if dtype is not None and dtype != code:
            raise ValueError("dtype %d does not match the gradient tensor's %s" % (dtype, grads.dtype))
        return code

    def set_params(self, x0) -> None:
        import torch
        self._check_tensor(x0, "x0", (self.n_padded,), (torch.float32,), "cuda")
        mtdao_set_params(self.h, self._ptr(x0))

    def step(self, grads, lr: float, sync_mask: int | None = None, dtype: int | None = None) -> int:
        """One local step; by default averages whatever is due at its end.
        Returns the sync mask that was applied."""
        if sync_mask is None:
            sync_mask = mtdao_sync_due(self.h)
        self._check_tensor(grads, "grads", (self.M, self.n_padded), self._grad_dtypes(), "cuda")
        dtype = self._grad_code(grads, dtype)
        mtdao_step(self.h, self._ptr(grads), dtype, lr, sync_mask)
        return sync_mask

    def step_host(self, grads_host, lr: float, sync_mask: int | None = None,
                  dtype: int | None = None) -> int:
        if sync_mask is None:
            sync_mask = mtdao_sync_due(self.h)
        self._check_tensor(grads_host, "grads_host", (self.M, self.n_padded), self._grad_dtypes(), "cpu")
        dtype = self._grad_code(grads_host, dtype)
        mtdao_step_host(self.h, self._ptr(grads_host), dtype, lr, sync_mask)
        return sync_mask

    def run(self, grads, lrs, dtype: int | None = None) -> None:
        """len(lrs) local steps in one call.  grads: a [count][M][n_padded]
        tensor (one buffer per step) or a [M][n_padded] tensor (or a raw
        device pointer to one) reused by every step."""
        three_d = not isinstance(grads, int) and grads.dim() == 3
        shape = (len(lrs), self.M, self.n_padded) if three_d else (self.M, self.n_padded)
        self._check_tensor(grads, "grads", shape, self._grad_dtypes(), "cuda")
        dtype = self._grad_code(grads, dtype)
        stride = grads.stride(0) * grads.element_size() if three_d else 0
        mtdao_run(self.h, self._ptr(grads), stride, dtype, lrs)

    def sync(self, mask: int) -> None:
        mtdao_sync(self.h, mask)

    def sync_due(self) -> int:
        return mtdao_sync_due(self.h)

    def sync_stats(self, mask: int):
        """Average the masked states and return their diagnostics as a
        device tensor [n_masked][2 + 2M] (see mtdao_sync_stats)."""
        import torch
        k = bin(mask).count("1")
        out = torch.empty((k, 2 + 2 * self.M), dtype=torch.float64, device="cuda")
        mtdao_sync_stats(self.h, mask, out.data_ptr())
        return out

    def track_anchor(self, state_mask: int = 1) -> None:
        """Keep anchors for the states in state_mask (bit 0 = x); 0 frees all."""
        mtdao_track_anchor(self.h, state_mask)

    def pseudo_grad_stats(self, state: int = 0):
        """Change diagnostics of one state against its anchor as a device
        tensor [2M + 2] (see mtdao_pseudo_grad_stats); state 0 gives the
        pseudo-gradients."""
        import torch
        out = torch.empty((2 * self.M + 2,), dtype=torch.float64, device="cuda")
        mtdao_pseudo_grad_stats(self.h, state, out.data_ptr())
        return out

    def tensor_views(self, flat, shapes):
        """Views of one flattened [n_padded] vector laid out like this
        handle's tensor list -- a replica's state (``state_view(s)[m]``) or a
        row of a gradient buffer -- one per tensor, shaped by ``shapes``
        (each with the numel given at construction).  The views share the
        vector's memory: a model can use a replica's parameters in place and
        write its gradients in place, with no packing copy."""
        import math
        if len(shapes) != len(self.numels):
            raise ValueError("expected %d shapes, got %d" % (len(self.numels), len(shapes)))
        views = []
        for off, k, shp in zip(self.offsets, self.numels, shapes):
            shp = tuple(int(d) for d in shp)
            if math.prod(shp) != k:
                raise ValueError("shape %s does not hold %d elements" % (shp, k))
            views.append(flat[off:off + k].view(shp))
        return views

    def state_ptr(self, state: int, replica: int) -> int:
        return mtdao_get_state_ptr(self.h, state, replica)

    def state_view(self, state: int):
        """Torch view [M][n_padded] (fp32, device) of one state across replicas."""
        import torch
        ptr = mtdao_get_state_ptr(self.h, state, 0)
        return _DevView.wrap(ptr, (self.M, self.n_padded))

    @property
    def t(self) -> int:
        return mtdao_get_step(self.h)

    @t.setter
    def t(self, value: int) -> None:
        mtdao_set_step(self.h, value)


class _DevView:
    """Zero-copy torch tensor over library-owned device memory (float32)."""

    @staticmethod
    def wrap(ptr: int, shape):
        import torch

        class _Cai:
            def __init__(self, p, shp):
                self.__cuda_array_interface__ = {
                    "shape": tuple(shp), "typestr": "<f4", "data": (p, False), "version": 3,
                    "strides": None}
        return torch.as_tensor(_Cai(ptr, shape), device="cuda")
