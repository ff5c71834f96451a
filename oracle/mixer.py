"""fp64 oracle of the steps either side of the scan in a Mamba mixer: the
causal depthwise convolution of width 4 (with SiLU) whose last three inputs
are part of the cached boundary state, the step size softplus(dt_raw + bias),
and the SiLU-gated output (Sec. 4, eq. prefix-cache; Sec. 4.1, eq. cache-c4:
the cache holds the convolution state and the state-space state; Appendix C:
convolution width 4).

TEST INFRASTRUCTURE, like the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and the CPU baseline of ``bench.py`` may use it.

Readings (the paper names these parts without writing them out):
  * One causal depthwise convolution per layer acts on the layer's forward
    input stream: pre_t = b + sum_{j=0..3} w[j] xr_{t-3+j} (tap 3 multiplies
    the current token), then x = SiLU(pre). A noisy block continues the
    convolution from the clean stream: window positions before the block's
    first token read the clean raw inputs there (the convolution part of the
    boundary state), positions inside the block read the noisy raw inputs.
    Positions before token 0 read the initial convolution state (zero unless
    given). Both scan directions of a noisy block read the convolved input.
  * dt = softplus(dt_raw + bias): bias_f for the clean stream and the noisy
    forward direction (the layer's forward scan), bias_r for the reverse one.
  * out = y * SiLU(z), with y the scan's output of the stream (both
    directions and skip terms for the noisy stream) and z the stream's gate.
  * The convolution state of boundary k is the clean raw input of the last
    three tokens of block k (tokens before 0 from the initial state).

Every function takes and returns fp64 numpy arrays; token-by-channel tensors
are [Bt, L, D], w [D, 4], b, bias_f, bias_r [D], convolution states
[Bt, 3, D] (oldest first). The scan steps call the pinned diagonal oracle.
Pins: tests/test_mixer_oracle_pins.py.
"""

from __future__ import annotations

import numpy as np

from . import active_block as _active_block
from . import backward as _backward
from . import boundary_states as _boundary_states
from . import forward as _forward

WIDTH = 4


def silu(z):
    z = np.asarray(z, np.float64)
    return z / (1.0 + np.exp(-z))


def dsilu(z):
    """d SiLU / dz = s (1 + z (1 - s)), s = sigmoid(z)."""
    z = np.asarray(z, np.float64)
    s = 1.0 / (1.0 + np.exp(-z))
    return s * (1.0 + z * (1.0 - s))


def softplus(z):
    z = np.asarray(z, np.float64)
    return np.maximum(z, 0.0) + np.log1p(np.exp(-np.abs(z)))


def sigmoid(z):
    return 1.0 / (1.0 + np.exp(-np.asarray(z, np.float64)))


def _windows(xr_c, xr_n, block, conv_init):
    """Raw inputs seen by tap j of every clean and noisy token: arrays
    [WIDTH, Bt, L, D] (tap j holds the input at position t - 3 + j)."""
    xr_c = np.asarray(xr_c, np.float64)
    Bt, L, D = xr_c.shape
    init = np.zeros((Bt, WIDTH - 1, D)) if conv_init is None else np.asarray(conv_init, np.float64)
    ext_c = np.concatenate([init, xr_c], axis=1)  # position u at index u + 3
    wc = np.stack([ext_c[:, j:j + L] for j in range(WIDTH)])
    wn = None
    if xr_n is not None:
        xr_n = np.asarray(xr_n, np.float64)
        wn = np.empty_like(wc)
        for t in range(L):
            k0 = (t // block) * block  # first token of the noisy block of t
            for j in range(WIDTH):
                u = t - (WIDTH - 1) + j
                wn[j, :, t] = xr_n[:, u] if u >= k0 else ext_c[:, u + WIDTH - 1]
    return wc, wn


def _conv(win, w, b):
    w = np.asarray(w, np.float64)
    return np.asarray(b, np.float64) + sum(w[:, j] * win[j] for j in range(WIDTH))


def prep(block, xr_c, dtr_c, xr_n, dtr_f, dtr_r, w, b, bias_f, bias_r, conv_init=None):
    """Scan inputs from the raw projections: returns a dict with pre_c, x_c,
    dt_c and (if xr_n is given) pre_n, x_n, dt_f, dt_r."""
    wc, wn = _windows(xr_c, xr_n, block, conv_init)
    o = {"pre_c": _conv(wc, w, b)}
    o["x_c"] = silu(o["pre_c"])
    o["dt_c"] = softplus(np.asarray(dtr_c, np.float64) + bias_f)
    if xr_n is not None:
        o["pre_n"] = _conv(wn, w, b)
        o["x_n"] = silu(o["pre_n"])
        o["dt_f"] = softplus(np.asarray(dtr_f, np.float64) + bias_f)
        o["dt_r"] = softplus(np.asarray(dtr_r, np.float64) + bias_r)
    o["_wc"], o["_wn"] = wc, wn
    return o


def forward(block, xr_c, dtr_c, B_c, C_c, z_c, xr_n, dtr_f, B_f, C_f, dtr_r, B_r, C_r, z_n,
            A_f, D_f, A_r, D_r, w, b, bias_f, bias_r):
    """All-block forward of the mixer. Returns (out_c, out_n, states)."""
    p = prep(block, xr_c, dtr_c, xr_n, dtr_f, dtr_r, w, b, bias_f, bias_r)
    y_c, y_n, st = _forward(block, p["x_c"], p["dt_c"], B_c, C_c, p["x_n"], p["dt_f"], B_f, C_f, p["dt_r"], B_r,
                            C_r, A_f, D_f, A_r, D_r)
    return y_c * silu(z_c), y_n * silu(z_n), st


def conv_states(block, xr_c, conv_init=None, emit_all=True):
    """Convolution part of the cache: the raw clean inputs of the last three
    tokens of every block ([Bt, L/Bs, 3, D]) or of the stream ([Bt, 1, 3, D])."""
    xr_c = np.asarray(xr_c, np.float64)
    Bt, L, D = xr_c.shape
    init = np.zeros((Bt, WIDTH - 1, D)) if conv_init is None else np.asarray(conv_init, np.float64)
    ext = np.concatenate([init, xr_c], axis=1)
    ends = range(block, L + 1, block) if emit_all else [L]
    return np.stack([ext[:, e:e + WIDTH - 1] for e in ends], axis=1)


def boundary_states(block, xr_c, dtr_c, B_c, C_c, A_f, D_f, w, b, bias_f, init_state=None, conv_init=None,
                    emit_all=True):
    """Cache build or append: (SSM states, convolution states)."""
    p = prep(block, xr_c, dtr_c, None, None, None, w, b, bias_f, bias_f, conv_init)
    st, _ = _boundary_states(block, p["x_c"], p["dt_c"], B_c, C_c, A_f, D_f, init_state, emit_all)
    return st, conv_states(block, xr_c, conv_init, emit_all)


def active_block(seed, conv_seed, xr_n, dtr_f, B_f, C_f, dtr_r, B_r, C_r, z_n, A_f, D_f, A_r, D_r,
                 w, b, bias_f, bias_r):
    """One noisy block from the cached SSM state and convolution state."""
    xr_n = np.asarray(xr_n, np.float64)
    Bt, Bs, D = xr_n.shape
    # the block's convolution reads the cached raw inputs before its first token
    ext = np.concatenate([np.asarray(conv_seed, np.float64), xr_n], axis=1)
    pre = _conv(np.stack([ext[:, j:j + Bs] for j in range(WIDTH)]), w, b)
    y = _active_block(seed, silu(pre), softplus(np.asarray(dtr_f, np.float64) + bias_f), B_f, C_f,
                      softplus(np.asarray(dtr_r, np.float64) + bias_r), B_r, C_r, A_f, D_f, A_r, D_r)
    return y * silu(z_n)


def backward(block, xr_c, dtr_c, B_c, C_c, z_c, xr_n, dtr_f, B_f, C_f, dtr_r, B_r, C_r, z_n,
             A_f, D_f, A_r, D_r, w, b, bias_f, bias_r, dout_c, dout_n, dstates=None):
    """Gradients of <dout_c, out_c> + <dout_n, out_n> + <dstates, states> by the
    chain rule through the gate, the pinned scan backward and the input steps.
    Returns a dict keyed like the arguments (xr_c, ..., bias_r)."""
    p = prep(block, xr_c, dtr_c, xr_n, dtr_f, dtr_r, w, b, bias_f, bias_r)
    y_c, y_n, st = _forward(block, p["x_c"], p["dt_c"], B_c, C_c, p["x_n"], p["dt_f"], B_f, C_f, p["dt_r"], B_r,
                            C_r, A_f, D_f, A_r, D_r)
    dout_c = np.asarray(dout_c, np.float64)
    dout_n = np.asarray(dout_n, np.float64)
    g = {"z_c": dout_c * y_c * dsilu(z_c), "z_n": dout_n * y_n * dsilu(z_n)}
    s = _backward(block, p["x_c"], p["dt_c"], B_c, C_c, p["x_n"], p["dt_f"], B_f, C_f, p["dt_r"], B_r, C_r,
                  A_f, D_f, A_r, D_r, st, dout_c * silu(z_c), dout_n * silu(z_n), dstates)
    for k in ("B_c", "C_c", "B_f", "C_f", "B_r", "C_r", "A_f", "D_f", "A_r", "D_r"):
        g[k] = s[k]
    # softplus: d dt / d dt_raw = sigmoid(dt_raw + bias)
    g["dtr_c"] = s["dt_c"] * sigmoid(np.asarray(dtr_c, np.float64) + bias_f)
    g["dtr_f"] = s["dt_f"] * sigmoid(np.asarray(dtr_f, np.float64) + bias_f)
    g["dtr_r"] = s["dt_r"] * sigmoid(np.asarray(dtr_r, np.float64) + bias_r)
    g["bias_f"] = (g["dtr_c"] + g["dtr_f"]).sum(axis=(0, 1))
    g["bias_r"] = g["dtr_r"].sum(axis=(0, 1))
    # convolution: pre-activation gradients, then each tap's input
    dpc = s["x_c"] * dsilu(p["pre_c"])
    dpn = s["x_n"] * dsilu(p["pre_n"])
    g["b"] = dpc.sum(axis=(0, 1)) + dpn.sum(axis=(0, 1))
    g["w"] = np.stack([(dpc * p["_wc"][j]).sum(axis=(0, 1)) + (dpn * p["_wn"][j]).sum(axis=(0, 1))
                       for j in range(WIDTH)], axis=1)
    w = np.asarray(w, np.float64)
    Bt, L, D = dpc.shape
    dxc = np.zeros((Bt, L, D))
    dxn = np.zeros((Bt, L, D))
    for t in range(L):
        k0 = (t // block) * block
        for j in range(WIDTH):
            u = t - (WIDTH - 1) + j
            if u < 0:
                continue
            dxc[:, u] += w[:, j] * dpc[:, t]
            if u >= k0:
                dxn[:, u] += w[:, j] * dpn[:, t]
            else:
                dxc[:, u] += w[:, j] * dpn[:, t]
    g["xr_c"], g["xr_n"] = dxc, dxn
    return g
