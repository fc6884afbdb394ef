"""Shared helpers of the GPU-vs-oracle parity tests.

Tolerance: for each state tensor r (oracle, fp64) and a (GPU, fp32) after
T steps

    err = max_i |a_i - r_i| / max(|r_i|, rms(r))  <=  1e-5

i.e. the relative error of every element, where an element smaller than the
tensor's RMS magnitude is judged against that RMS (a value that cancels
towards zero carries the rounding error of the larger operands it came
from).  Positions of NaN/Inf must agree.  Beside it ``compare`` reports the
raw relative error max |a_i - r_i| / |r_i| over the elements with r_i != 0
(no floor), which shows how much the floor absorbs near zero crossings; the
bar applies to the floored figure.  The bar is 1e-5; the fp32 path
rounds every stored state once per step plus a few operations (a few
units of 2^-24 relative), the EMAs contract, and errors grow at most like
a random walk over T steps, so measured errors stay near 1e-6.
"""
from __future__ import annotations

import numpy as np

from oracle.oracle import Oracle
from synth import generators as G
from synth import workloads as W

TOL = 1e-5
STATE_NAMES_CACHE = {}


def state_names(opt: dict):
    names = ["x"] + ["u%d" % (j + 1) for j in range(opt["n_mom"])]
    if opt["base"] != "sgdm":
        names.append("v")
    return names


def rel_err(a, r) -> float:
    a = np.asarray(a, np.float64)
    r = np.asarray(r, np.float64)
    fa, fr = np.isfinite(a), np.isfinite(r)
    assert np.array_equal(fa, fr), "non-finite positions differ"
    a, r = a[fr], r[fr]
    if r.size == 0:
        return 0.0
    floor = float(np.sqrt(np.mean(r * r)))
    if floor == 0.0:
        return float(np.max(np.abs(a - r)))
    return float(np.max(np.abs(a - r) / np.maximum(np.abs(r), floor)))


def raw_rel_err(a, r) -> float:
    """max |a_i - r_i| / |r_i| over the finite elements with r_i != 0."""
    a = np.asarray(a, np.float64)
    r = np.asarray(r, np.float64)
    keep = np.isfinite(r) & np.isfinite(a) & (r != 0)
    if not keep.any():
        return 0.0
    return float(np.max(np.abs(a[keep] - r[keep]) / np.abs(r[keep])))


LAST_REPORT = {}


def oracle_run(opt, M, idx, T, lay, w, seed_grad, seed_init, lr=None, t0=0):
    """Run the oracle on the padded indices idx (all M workers) for T steps."""
    lr = opt.get("lr", 1e-3) if lr is None else lr
    idx = np.asarray(idx, np.int64)
    x0 = G.init_params(w, lay, seed_init, idx).astype(np.float64)
    o = Oracle(opt, M, idx.size, x0=x0)
    for t in range(t0, t0 + T):
        g = np.stack([G.grads(w, lay, seed_grad, m, t, idx) for m in range(M)]).astype(np.float64)
        o.step(t, lr, g)
    o.settle(t0 + T)
    return o.states()


def compare(gpu_states: dict, ora_states: dict, tol=TOL):
    """Assert every state within tol (floored relative error); returns the
    floored errors per state.  The raw (unfloored) errors are kept in
    LAST_REPORT[state] = (floored, raw) and shown in the failure message."""
    errs = {k: rel_err(gpu_states[k], ora_states[k]) for k in ora_states}
    raw = {k: raw_rel_err(gpu_states[k], ora_states[k]) for k in ora_states}
    LAST_REPORT.clear()
    LAST_REPORT.update({k: (errs[k], raw[k]) for k in errs})
    bad = {k: e for k, e in errs.items() if not e <= tol}
    assert not bad, "parity errors above %g: %s (all: %s; raw |a-r|/|r|: %s)" % (tol, bad, errs, raw)
    return errs


def workload_dict(shapes, M, base="adam", betas=(0.9, 0.999), omega=None, beta2=0.999, eps=1e-8,
                  bias=None, clip="none", rho=1.0, px=4, pu=4, pv=4, phase="alg1", lr=1e-3,
                  grad_kind="normal", sigma=0.01, gdt="f32"):
    n = len(betas)
    if omega is None:
        omega = [0.95 / n] * n
    if bias is None:
        bias = base == "adam"
    pu_list = list(pu) if isinstance(pu, (list, tuple)) else [pu] * n
    opt = {"base": base, "n_mom": n, "beta1": list(betas), "omega": list(omega), "beta2": beta2,
           "eps": eps, "bias_correction": bias, "clip_mode": clip, "clip_rho": rho,
           "period_x": px, "period_u": pu_list, "period_v": pv, "sync_phase": phase, "lr": lr}
    return {"name": "custom", "shapes": list(shapes), "M": M, "grad_kind": grad_kind,
            "grad_sigma": sigma, "grad_dtype": gdt, "init_sigma": 0.02, "opt": opt}


def host_grads(w, lay, seed, t, idx):
    return np.stack([G.grads(w, lay, seed, m, t, idx) for m in range(w["M"])])


def sample_indices(lay, count, seed=0):
    """Sampled padded indices: random positions plus every tensor's first and
    last 8 elements and the last elements of the padded vector."""
    rng = np.random.default_rng(seed)
    n = lay["n_padded"]
    pts = [rng.integers(0, n, size=count)]
    for off, num in zip(lay["offsets"], lay["numels"]):
        pts.append(np.arange(off, off + min(8, num)))
        pts.append(np.arange(off + max(num - 8, 0), off + num))
    pts.append(np.arange(n - 16, n))
    return np.unique(np.concatenate(pts)).astype(np.int64)
