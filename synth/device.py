"""GPU side of the synthetic input generator (``synth_dev.cu``).

Fills device buffers with the same values ``generators.py`` computes on the
host, so full-size gradients never cross the host link.  Built in-tree with
nvcc for sm_103a; loading fails loudly if the library is missing.
"""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "synth_dev.cu")
LIB = os.path.join(HERE, "_build", "libmtdao_synth.so")
KIND_IDS = {"normal": 0, "student_t3": 1, "normal_outliers": 2}
_lib = None


def build(force: bool = False) -> str:
    import fcntl

    def fresh():
        return os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC)

    if not force and fresh():
        return LIB
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    with open(os.path.join(os.path.dirname(LIB), ".lock"), "w") as lock:
        fcntl.flock(lock, fcntl.LOCK_EX)           # one builder at a time
        if force or not fresh():
            nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
            tmp = LIB + ".%d.tmp" % os.getpid()
            cmd = [nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17",
                   "-Xcompiler", "-fPIC", "-shared", SRC, "-o", tmp, "-lcudart"]
            subprocess.run(cmd, check=True)
            os.replace(tmp, LIB)
    return LIB


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise ImportError("libmtdao_synth.so is not built; run synth.device.build()")
        lib = ctypes.CDLL(LIB)
        lib.synth_fill.restype = ctypes.c_int
        lib.synth_fill.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_uint64,
                                   ctypes.c_uint64, ctypes.c_int, ctypes.c_int64, ctypes.c_int64,
                                   ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                   ctypes.c_void_p]
        lib.synth_toy_grad.restype = ctypes.c_int
        lib.synth_toy_grad.argtypes = [ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                       ctypes.c_int64, ctypes.c_int64, ctypes.c_uint64, ctypes.c_int64,
                                       ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p]
        _lib = lib
    return _lib


class DeviceInputs:
    """Generates a workload's gradients and initial parameters on the GPU."""

    def __init__(self, workload: dict, layout: dict, seed_grad: int, seed_init: int):
        import torch
        self.w = workload
        self.lay = layout
        self.seed_grad = int(seed_grad)
        self.seed_init = int(seed_init)
        self.n = int(layout["n_padded"])
        # zero-size tensors own no element; the device search skips them
        keep = [(o, k) for o, k in zip(layout["offsets"], layout["numels"]) if k > 0]
        self.off = torch.tensor([o for o, _ in keep], dtype=torch.int64, device="cuda")
        self.num = torch.tensor([k for _, k in keep], dtype=torch.int64, device="cuda")
        self.n_tensors = len(keep)
        self.lib = _load()

    def _fill(self, out, bf16, kind, seed, stream_id, M, t, sigma):
        import torch
        st = torch.cuda.current_stream().cuda_stream
        rc = self.lib.synth_fill(ctypes.c_void_p(out.data_ptr()), int(bf16), int(kind), seed, stream_id,
                                 M, self.n, int(t), ctypes.c_float(sigma),
                                 ctypes.c_void_p(self.off.data_ptr()), ctypes.c_void_p(self.num.data_ptr()),
                                 self.n_tensors, ctypes.c_void_p(st))
        if rc != 0:
            raise RuntimeError("synth_fill failed with CUDA error %d" % rc)

    def grads(self, t: int, out=None):
        """Gradient buffer [M][n_padded] for step t (float32 or bfloat16)."""
        import torch
        bf16 = self.w.get("grad_dtype", "f32") == "bf16"
        M = self.w["M"]
        if out is None:
            out = torch.empty((M, self.n), dtype=torch.bfloat16 if bf16 else torch.float32,
                              device="cuda")
        self._fill(out, bf16, KIND_IDS[self.w["grad_kind"]], self.seed_grad, 1, M, t,
                   float(self.w["grad_sigma"]))
        return out

    def init_params(self, out=None):
        import torch
        if out is None:
            out = torch.empty((self.n,), dtype=torch.float32, device="cuda")
        self._fill(out, False, 0, self.seed_init, 2, 1, 0, float(self.w.get("init_sigma", 0.02)))
        return out


TOY_KINDS = {"quadratic": 0, "rosenbrock": 1}


def toy_grad(kind: str, x_ptr: int, g, M: int, n_padded: int, n_real: int, seed: int, t: int,
             sigma: float, lam=None) -> None:
    """Noisy toy-objective gradient of the workers' parameters at device
    pointer x_ptr ([M][n_padded] fp32) into the float32 tensor g."""
    import torch
    lib = _load()
    st = torch.cuda.current_stream().cuda_stream
    rc = lib.synth_toy_grad(TOY_KINDS[kind], ctypes.c_void_p(x_ptr), ctypes.c_void_p(g.data_ptr()), M,
                            n_padded, n_real, seed, int(t), ctypes.c_float(sigma),
                            ctypes.c_void_p(lam.data_ptr() if lam is not None else 0), ctypes.c_void_p(st))
    if rc != 0:
        raise RuntimeError("synth_toy_grad failed with CUDA error %d" % rc)
