"""Shared helpers of the GPU parity tests: run the CUDA path and the oracle on
the same seeded inputs and compare them element by element.

Tolerance: per tensor, max_i (|gpu_i - oracle_i| - u |oracle_i|) <= tol * max_i |oracle_i|
with tol = 2e-3 for forward outputs and 5e-3 for gradients (the stated
bounds for bf16 inputs with fp32 accumulation), and u the unit roundoff of
the output storage type (2^-8 for bf16 outputs, 0 for fp32 outputs): a bf16
output cannot be closer to the exact value than its own rounding.
"""

from __future__ import annotations

import os

import numpy as np

FWD_TOL = 2e-3
GRAD_TOL = 5e-3
BF16_U = 2.0 ** -8

FWD_NAMES = ("x_c", "dt_c", "B_c", "C_c", "x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r",
             "A_f", "D_f", "A_r", "D_r")
PARAMS = ("A_f", "D_f", "A_r", "D_r")


def rel_err(gpu, ora, u=0.0):
    gpu = np.asarray(gpu, dtype=np.float64)
    ora = np.asarray(ora, dtype=np.float64)
    scale = float(np.max(np.abs(ora))) if ora.size else 0.0
    if scale == 0.0:
        return float(np.max(np.abs(gpu))) if gpu.size else 0.0
    excess = np.abs(gpu - ora) - u * np.abs(ora)
    return float(max(0.0, np.max(excess)) / scale)


def elementwise_rel_err(gpu, ora):
    """Largest per-element relative error |gpu - oracle| / (|oracle| + 1e-3 rms(oracle)):
    reported for information next to the per-tensor bound (the rms term keeps
    elements near zero from dominating)."""
    gpu = np.asarray(gpu, dtype=np.float64)
    ora = np.asarray(ora, dtype=np.float64)
    if ora.size == 0:
        return 0.0
    rms = float(np.sqrt(np.mean(ora * ora)))
    if rms == 0.0:
        return float(np.max(np.abs(gpu)))
    return float(np.max(np.abs(gpu - ora) / (np.abs(ora) + 1e-3 * rms)))


# (test id, tensor, per-tensor error, elementwise error) of every comparison
# made in this process, printed in the pytest summary
RECORD = []
_CURRENT_TEST = [""]


def assert_close(name, gpu, ora, tol, u=0.0):
    e = rel_err(gpu, ora, u)
    RECORD.append((_CURRENT_TEST[0], name, e, elementwise_rel_err(gpu, ora)))
    assert e <= tol, f"{name}: relative error {e:.3e} above {tol:.1e}"
    return e


def oracle_threads():
    import oracle
    oracle.set_threads(max(1, min(16, os.cpu_count() or 1)))


def oracle_forward(wl, sub=None):
    """Oracle forward on the workload, optionally restricted to channels `sub`."""
    import oracle
    d = slice_channels(wl, sub)
    return oracle.forward(wl.block, *[d[k] for k in FWD_NAMES])


def oracle_backward(wl, states, use_dy_c=True, use_dstates=False, sub=None):
    """`states` are the oracle's states of the (possibly channel-sliced) problem."""
    import oracle
    d = slice_channels(wl, sub)
    return oracle.backward(wl.block, *[d[k] for k in FWD_NAMES], states, d["dy_c"] if use_dy_c else None,
                           d["dy_n"], d["dstates"] if use_dstates else None)


def slice_channels(wl, sub):
    """fp64 inputs of the workload; with `sub`, only those channels (d indices).
    Channels are independent in every output except the sums over channels
    (dB, dC), so a channel slice reproduces the full problem's per-channel
    outputs and the parameter gradients of those channels exactly."""
    out = {}
    for k in wl.t32:
        a = wl.t32[k]
        if sub is not None:
            if k in ("A_f", "A_r", "D_f", "D_r"):
                a = a[sub]
            elif k == "dstates":
                a = a[:, :, sub]
            elif k == "init_state":
                a = a[:, sub]
            elif a.ndim == 3 and k not in ("B_c", "C_c", "B_f", "C_f", "B_r", "C_r"):
                a = a[:, :, sub]
        out[k] = np.ascontiguousarray(a, dtype=np.float64)
    return out
