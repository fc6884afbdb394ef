"""ctypes front end of the plain C oracle (``mtdao_oracle.c``).

TEST INFRASTRUCTURE ONLY.  The oracle is the slow, obviously correct
reference that the CUDA library is checked against.  Only the test suite,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may
import this module.  It never imports the CUDA library and the CUDA library
never imports it.

The oracle holds every state in fp64 and follows the paper's Algorithm 1
(MT-DAO-Adam), Algorithm 2 (MT-DAO-ADOPT) and Algorithm 3 (MT-DAO-SGDM) in the
order they are written.  Configurations are the plain dictionaries described
in ``synth.workloads`` (base, n_mom, beta1, omega, beta2, eps, ...).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mtdao_oracle.c")
_LIB = os.path.join(_HERE, "_build", "liboracle.so")
_MAX_MOM = 8
_lock = threading.Lock()
_lib = None

BASES = {"adam": 0, "adopt": 1, "sgdm": 2}
CLIPS = {"none": 0, "global_norm": 1, "elementwise": 2}
PHASES = {"alg1": 0, "alg2_literal": 1}


class _Cfg(ctypes.Structure):
    _fields_ = [
        ("base", ctypes.c_int),
        ("n_mom", ctypes.c_int),
        ("beta1", ctypes.c_double * _MAX_MOM),
        ("omega", ctypes.c_double * _MAX_MOM),
        ("beta2", ctypes.c_double),
        ("eps", ctypes.c_double),
        ("bias_correction", ctypes.c_int),
        ("clip_mode", ctypes.c_int),
        ("clip_rho", ctypes.c_double),
        ("period_x", ctypes.c_longlong),
        ("period_u", ctypes.c_longlong * _MAX_MOM),
        ("period_v", ctypes.c_longlong),
        ("sync_phase", ctypes.c_int),
        ("adopt_prev_v", ctypes.c_int),
    ]


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no FMA contraction, no fast-math)."""
    import fcntl
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)

    def fresh():
        return os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)

    if not force and fresh():
        return _LIB
    with open(os.path.join(os.path.dirname(_LIB), ".lock"), "w") as lock:
        fcntl.flock(lock, fcntl.LOCK_EX)           # one builder at a time
        if force or not fresh():
            tmp = _LIB + ".%d.tmp" % os.getpid()
            cmd = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-ffp-contract=off",
                   "-fno-fast-math", _SRC, "-o", tmp, "-lm"]
            subprocess.run(cmd, check=True)
            os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            dp = ctypes.POINTER(ctypes.c_double)
            cp = ctypes.POINTER(_Cfg)
            lib.mto_step.argtypes = [cp, ctypes.c_int, ctypes.c_longlong, ctypes.c_longlong,
                                     ctypes.c_double, dp, dp, dp, dp]
            lib.mto_step.restype = ctypes.c_int
            lib.mto_sync.argtypes = [cp, ctypes.c_int, ctypes.c_longlong, ctypes.c_uint,
                                     dp, dp, dp]
            lib.mto_sync.restype = None
            lib.mto_settle.argtypes = [cp, ctypes.c_int, ctypes.c_longlong, ctypes.c_longlong,
                                       dp, dp, dp]
            lib.mto_settle.restype = None
            lib.mto_run.argtypes = [cp, ctypes.c_int, ctypes.c_longlong, ctypes.c_longlong,
                                    ctypes.c_longlong, dp, dp, dp, dp, dp]
            lib.mto_run.restype = ctypes.c_int
            lib.mto_due_before_step.argtypes = [cp, ctypes.c_longlong]
            lib.mto_due_before_step.restype = ctypes.c_uint
            lib.mto_due_after_step.argtypes = [cp, ctypes.c_longlong]
            lib.mto_due_after_step.restype = ctypes.c_uint
            lib.mto_num_states.argtypes = [cp]
            lib.mto_num_states.restype = ctypes.c_int
            lib.mto_grad_norm.argtypes = [ctypes.c_longlong, dp]
            lib.mto_grad_norm.restype = ctypes.c_double
            lib.mto_adopt_clip_bound.argtypes = [ctypes.c_longlong]
            lib.mto_adopt_clip_bound.restype = ctypes.c_double
            lib.mto_mean_over_workers.argtypes = [ctypes.c_int, ctypes.c_longlong, dp]
            lib.mto_mean_over_workers.restype = None
            lib.mto_state_stats.argtypes = [ctypes.c_int, ctypes.c_longlong, dp, dp]
            lib.mto_state_stats.restype = None
            lib.mto_pseudo_grad_stats.argtypes = [ctypes.c_int, ctypes.c_longlong, dp, dp, dp]
            lib.mto_pseudo_grad_stats.restype = None
            lib.mto_half_life.argtypes = [ctypes.c_double]
            lib.mto_half_life.restype = ctypes.c_double
            lib.mto_half_life_periods.argtypes = [cp, ctypes.c_longlong]
            lib.mto_half_life_periods.restype = None
            lib.mto_comm_reduction.argtypes = [cp]
            lib.mto_comm_reduction.restype = ctypes.c_double
            _lib = lib
    return _lib


def make_cfg(cfg: dict) -> _Cfg:
    """Translate a workload dictionary into the oracle's C struct."""
    c = _Cfg()
    n = int(cfg["n_mom"])
    c.base = BASES[cfg["base"]]
    c.n_mom = n
    for j in range(n):
        c.beta1[j] = float(cfg["beta1"][j])
        c.omega[j] = float(cfg["omega"][j])
        c.period_u[j] = int(cfg["period_u"][j])
    c.beta2 = float(cfg.get("beta2", 0.999))
    c.eps = float(cfg.get("eps", 1e-8))
    c.bias_correction = 1 if cfg.get("bias_correction", True) else 0
    c.clip_mode = CLIPS[cfg.get("clip_mode", "none")]
    c.clip_rho = float(cfg.get("clip_rho", 1.0))
    c.period_x = int(cfg["period_x"])
    c.period_v = int(cfg.get("period_v", 0))
    c.sync_phase = PHASES[cfg.get("sync_phase", "alg1")]
    c.adopt_prev_v = 1 if cfg.get("adopt_prev_v", False) else 0
    return c


def _ptr(a: np.ndarray):
    assert a.dtype == np.float64 and a.flags.c_contiguous
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


class Oracle:
    """M workers' states for n elements, held in fp64.

    Layout: ``x[M][n]``, ``u[N][M][n]``, ``v[M][n]`` (``v`` unused for SGDM).
    """

    def __init__(self, cfg: dict, M: int, n: int, x0=None):
        self.cfg = dict(cfg)
        self.c = make_cfg(cfg)
        self.lib = _load()
        self.M, self.n, self.N = int(M), int(n), int(cfg["n_mom"])
        self.x = np.zeros((self.M, self.n), np.float64)
        self.u = np.zeros((self.N, self.M, self.n), np.float64)
        self.v = np.zeros((self.M, self.n), np.float64)
        if x0 is not None:
            self.x[:] = np.asarray(x0, np.float64)[None, :]

    def step(self, t: int, lr: float, g: np.ndarray) -> None:
        """Iteration t for all workers; g is ``[M][n]``."""
        g = np.ascontiguousarray(g, np.float64).reshape(self.M, self.n)
        rc = self.lib.mto_step(ctypes.byref(self.c), self.M, self.n, int(t), float(lr),
                               _ptr(g), _ptr(self.x), _ptr(self.u), _ptr(self.v))
        if rc != 0:
            raise ValueError("oracle rejected the configuration")

    def settle(self, t: int) -> None:
        """Apply the averages that iteration t would read (Algorithm 1 rule)."""
        self.lib.mto_settle(ctypes.byref(self.c), self.M, self.n, int(t),
                            _ptr(self.x), _ptr(self.u), _ptr(self.v))

    def sync(self, mask: int) -> None:
        self.lib.mto_sync(ctypes.byref(self.c), self.M, self.n, int(mask),
                          _ptr(self.x), _ptr(self.u), _ptr(self.v))

    def due_before_step(self, t: int) -> int:
        return int(self.lib.mto_due_before_step(ctypes.byref(self.c), int(t)))

    def due_after_step(self, t: int) -> int:
        return int(self.lib.mto_due_after_step(ctypes.byref(self.c), int(t)))

    def num_states(self) -> int:
        return int(self.lib.mto_num_states(ctypes.byref(self.c)))

    def states(self) -> dict:
        """Named copies of the states: x, u1..uN and (Adam/ADOPT) v."""
        out = {"x": self.x.copy()}
        for j in range(self.N):
            out["u%d" % (j + 1)] = self.u[j].copy()
        if self.cfg["base"] != "sgdm":
            out["v"] = self.v.copy()
        return out


def run(cfg: dict, M: int, n: int, t0: int, lrs, g, x, u, v) -> None:
    """T iterations in one C call (timing helper); arrays updated in place."""
    lib = _load()
    c = make_cfg(cfg)
    lrs = np.ascontiguousarray(lrs, np.float64)
    g = np.ascontiguousarray(g, np.float64)
    rc = lib.mto_run(ctypes.byref(c), int(M), int(n), int(t0), int(lrs.shape[0]),
                     _ptr(lrs), _ptr(g), _ptr(x), _ptr(u), _ptr(v))
    if rc != 0:
        raise ValueError("oracle rejected the configuration")


def grad_norm(g: np.ndarray) -> float:
    g = np.ascontiguousarray(g, np.float64).ravel()
    return float(_load().mto_grad_norm(g.size, _ptr(g)))


def adopt_clip_bound(t: int) -> float:
    return float(_load().mto_adopt_clip_bound(int(t)))


def state_stats(s: np.ndarray) -> np.ndarray:
    """Cross-worker diagnostics of an ``[M][n]`` state (see mto_state_stats):
    [variance, ||mean||^2, ||s_m||^2 (M), <s_m, mean> (M)]."""
    s = np.ascontiguousarray(s, np.float64)
    M = s.shape[0]
    out = np.zeros(2 + 2 * M, np.float64)
    _load().mto_state_stats(M, s.size // M, _ptr(s), _ptr(out))
    return out


def pseudo_grad_stats(x: np.ndarray, anchor: np.ndarray) -> np.ndarray:
    """Pseudo-gradient diagnostics of the workers' parameters x ``[M][n]``
    against the round's starting point ``anchor`` ``[n]`` (see
    mto_pseudo_grad_stats): [||x_m - a||^2 (M), <x_m - a, x_bar - a> (M),
    ||x_bar - a||^2, ||a||^2]."""
    x = np.ascontiguousarray(x, np.float64)
    a = np.ascontiguousarray(anchor, np.float64).ravel()
    M = x.shape[0]
    out = np.zeros(2 * M + 2, np.float64)
    _load().mto_pseudo_grad_stats(M, a.size, _ptr(x), _ptr(a), _ptr(out))
    return out


def mean_over_workers(s: np.ndarray) -> np.ndarray:
    """E_m over axis 0 of an ``[M][n]`` array (returns a new array)."""
    s = np.array(s, np.float64, order="C", copy=True)
    M = s.shape[0]
    lib = _load()
    lib.mto_mean_over_workers(M, s.size // M, _ptr(s))
    return s


def half_life(beta: float) -> float:
    """tau_0.5(beta) = ln 0.5 / ln beta (section 2.1)."""
    return float(_load().mto_half_life(float(beta)))


def half_life_periods(cfg: dict, period_x: int) -> dict:
    """The half-life sync strategy (see mto_half_life_periods): a copy of
    cfg with period_x, period_u and period_v set."""
    c = make_cfg(cfg)
    _load().mto_half_life_periods(ctypes.byref(c), int(period_x))
    out = dict(cfg)
    out["period_x"] = int(c.period_x)
    out["period_u"] = [int(c.period_u[j]) for j in range(int(cfg["n_mom"]))]
    out["period_v"] = int(c.period_v)
    return out


def comm_reduction(cfg: dict) -> float:
    """Communication saving over DDP (see mto_comm_reduction)."""
    c = make_cfg(cfg)
    return float(_load().mto_comm_reduction(ctypes.byref(c)))
