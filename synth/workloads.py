"""Synthetic workloads: parameter-list shapes and hyper-parameters.

Plain data shared by the tests and the benchmark.  The parameter lists stand
in for the paper's GPT-style models (Table of model architectures: peri-norm
decoders, vocabulary 50K, init sigma 0.02); no dataset or trained weight is
involved.  Tensor order for a decoder list: embedding [V*d], then per block
[qkv d*3d, proj d*d, fc1 d*F, fc2 F*d, ln1.w d, ln1.b d, ln2.w d, ln2.b d],
then final norm [d, d].

Hyper-parameters the paper leaves open are chosen as follows:
* omega_j = 0.95 / N for every j (the paper's N=1 runs use omega_1 = 0.95).
* The ADOPT workload has beta_1 = (0.95, 0.999) and beta_2 = 0.9999; the
  1B workload reuses the GPT-2-small betas (0.5, 0.9, 0.999).
* No gradient clipping in the listed workloads (they name none); clipping is
  exercised by separate test cases.

Layout convention (shared with the library, which computes it on its own):
each tensor starts at a multiple of 8 elements (32 B of fp32, 16 B of bf16)
and the per-worker length ``n_padded`` is rounded up to a multiple of 256
elements (1 KiB) so every worker's slab starts 1024-byte aligned.
"""
from __future__ import annotations

import copy

VOCAB = 50257
INIT_SEED = 20251005
GRAD_SEED = INIT_SEED + 1
TENSOR_ALIGN = 8
SLAB_ALIGN = 256


def decoder_shapes(vocab: int, d: int, ffn: int, blocks: int) -> list[int]:
    sizes = [vocab * d]
    for _ in range(blocks):
        sizes += [d * 3 * d, d * d, d * ffn, ffn * d, d, d, d, d]
    sizes += [d, d]
    return sizes


def layout(numels) -> dict:
    """Padded offsets of a flattened multi-tensor list (see module doc)."""
    offsets, pos = [], 0
    for k in numels:                       # zero-size tensors take no space
        offsets.append(pos)
        pos += (int(k) + TENSOR_ALIGN - 1) // TENSOR_ALIGN * TENSOR_ALIGN
    n_padded = (pos + SLAB_ALIGN - 1) // SLAB_ALIGN * SLAB_ALIGN
    return {"offsets": offsets, "numels": [int(k) for k in numels], "n_padded": n_padded}


def _opt(base, betas, beta2, lr, period_x, period_u, period_v, bias=True, clip="none"):
    n = len(betas)
    return {
        "base": base,
        "n_mom": n,
        "beta1": list(betas),
        "omega": [0.95 / n] * n,
        "beta2": beta2,
        "eps": 1e-8,
        "bias_correction": bias,
        "clip_mode": clip,
        "clip_rho": 1.0,
        "period_x": period_x,
        "period_u": [period_u] * n,
        "period_v": period_v,
        "sync_phase": "alg1",
        "lr": lr,
    }


WORKLOADS = {
    "tiny": {
        "name": "tiny",
        "desc": "flat fp32 vector n=1,048,576, M=4, N=2 beta=(0.9,0.999), Adam, "
                "grads N(0,1)*0.01, T=64, H=16",
        "shapes": [1 << 20],
        "M": 4,
        "T": 64,
        "grad_kind": "normal",
        "grad_sigma": 0.01,
        "grad_dtype": "f32",
        "init_sigma": 0.02,
        "opt": _opt("adam", (0.9, 0.999), 0.999, 1e-3, 16, 16, 16),
    },
    "gpt2_small": {
        "name": "gpt2_small",
        "desc": "GPT-2-small-shaped list (123,570,432 fp32, 99 tensors), M=4, N=3 "
                "beta=(0.5,0.9,0.999), Adam, grads Student-t(3)*1e-3, T=256, H=32",
        "shapes": decoder_shapes(VOCAB, 768, 3072, 12),
        "M": 4,
        "T": 256,
        "grad_kind": "student_t3",
        "grad_sigma": 1e-3,
        "grad_dtype": "f32",
        "init_sigma": 0.02,
        "opt": _opt("adam", (0.5, 0.9, 0.999), 0.999, 1e-3, 32, 32, 32),
    },
    "decoder_350m": {
        "name": "decoder_350m",
        "desc": "~350M decoder list (353,553,408, 24 blocks d=1024 FFN 4096), M=8, N=2 "
                "beta=(0.95,0.999), ADOPT beta2=0.9999, bf16 grads N(0,1e-3), "
                "H_x=64, H_u=H_v=16, T=512",
        "shapes": decoder_shapes(VOCAB, 1024, 4096, 24),
        "M": 8,
        "T": 512,
        "grad_kind": "normal",
        "grad_sigma": 1e-3,
        "grad_dtype": "bf16",
        "init_sigma": 0.02,
        "opt": _opt("adopt", (0.95, 0.999), 0.9999, 2.0 ** -8, 64, 16, 16, bias=False),
    },
    "decoder_1b": {
        "name": "decoder_1b",
        "desc": "~1B decoder list (1,311,086,592, 24 blocks d=2048 FFN 8192), M=4, N=3 "
                "beta=(0.5,0.9,0.999), Adam, grads N(0,1e-3) with 1% outliers x100, "
                "T=128, H=32",
        "shapes": decoder_shapes(VOCAB, 2048, 8192, 24),
        "M": 4,
        "T": 128,
        "grad_kind": "normal_outliers",
        "grad_sigma": 1e-3,
        "grad_dtype": "f32",
        "init_sigma": 0.02,
        "opt": _opt("adam", (0.5, 0.9, 0.999), 0.999, 1e-3, 32, 32, 32),
    },
    "profile_small": {
        "name": "profile_small",
        "desc": "flat fp32 vector n=2^25 with the ~1B workload's optimizer (M=4, N=3 "
                "beta=(0.5,0.9,0.999), Adam, grads N(0,1e-3) with 1% outliers x100, H=32): "
                "the same kernels on ~3 GB of device memory, for profiler captures",
        "shapes": [1 << 25],
        "M": 4,
        "T": 64,
        "grad_kind": "normal_outliers",
        "grad_sigma": 1e-3,
        "grad_dtype": "f32",
        "init_sigma": 0.02,
        "opt": _opt("adam", (0.5, 0.9, 0.999), 0.999, 1e-3, 32, 32, 32),
    },
    "profile_small_m16": {
        "name": "profile_small_m16",
        "desc": "flat fp32 vector n=2^23 with M=16 replicas and the ~1B workload's optimizer "
                "(N=3 beta=(0.5,0.9,0.999), Adam, grads N(0,1e-3) with 1% outliers x100, "
                "H=32): the block-staged fused step and one-pass diagnostics on ~3 GB of "
                "device memory, for profiler captures",
        "shapes": [1 << 23],
        "M": 16,
        "T": 64,
        "grad_kind": "normal_outliers",
        "grad_sigma": 1e-3,
        "grad_dtype": "f32",
        "init_sigma": 0.02,
        "opt": _opt("adam", (0.5, 0.9, 0.999), 0.999, 1e-3, 32, 32, 32),
    },
    "profile_small_adopt": {
        "name": "profile_small_adopt",
        "desc": "flat vector n=2^24 with the ~350M workload's optimizer (M=8, N=2 "
                "beta=(0.95,0.999), ADOPT beta2=0.9999, bf16 grads N(0,1e-3), H_x=64, "
                "H_u=H_v=16): the same kernels on ~2.4 GB of device memory, for profiler captures",
        "shapes": [1 << 24],
        "M": 8,
        "T": 64,
        "grad_kind": "normal",
        "grad_sigma": 1e-3,
        "grad_dtype": "bf16",
        "init_sigma": 0.02,
        "opt": _opt("adopt", (0.95, 0.999), 0.9999, 2.0 ** -8, 64, 16, 16, bias=False),
    },
}

SWEEP_BETAS = (0.9, 0.999, 0.5, 0.99)


def sweep_point(log2_n: int, M: int, N: int, H: int, base: str = "adam") -> dict:
    """One point of the flat-vector sweep (n = 2**log2_n)."""
    opt = _opt(base, SWEEP_BETAS[:N], 0.999 if base != "adopt" else 0.9999,
               1e-3, H, H, H, bias=(base == "adam"))
    if N == 1 and H == 1:
        opt["omega"] = [1.0]        # base-optimizer reduction point
    return {
        "name": "sweep_n%d_M%d_N%d_H%d" % (log2_n, M, N, H),
        "desc": "flat fp32 n=2^%d, M=%d, N=%d, H=%d" % (log2_n, M, N, H),
        "shapes": [1 << log2_n],
        "M": M,
        "T": 3 * H if H > 1 else 8,
        "grad_kind": "normal",
        "grad_sigma": 0.01,
        "grad_dtype": "f32",
        "init_sigma": 0.02,
        "opt": opt,
    }


def get(name: str) -> dict:
    return copy.deepcopy(WORKLOADS[name])


def bytes_per_step(w: dict) -> int:
    """Algorithmic HBM bytes of one local step: every state read and written
    once, the gradient read once."""
    n = layout(w["shapes"])["n_padded"]
    N = w["opt"]["n_mom"]
    states = 1 + N + (0 if w["opt"]["base"] == "sgdm" else 1)
    gb = 2 if w.get("grad_dtype") == "bf16" else 4
    return w["M"] * n * (8 * states + gb)


def bytes_per_sync(w: dict, n_states: int) -> int:
    n = layout(w["shapes"])["n_padded"]
    return 8 * w["M"] * n * n_states
