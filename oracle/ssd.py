"""fp64 oracle for the Mamba-2 (SSD) form of the block-restricted bidirectional scan.

TEST INFRASTRUCTURE, like the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and the CPU baseline of ``bench.py`` may use it.

The paper's trained mixers are Mamba-2 layers (Appendix C: state size 64 or
128, chunk 128; block 256). In that form the decay is one
scalar per head, A[h], and B_t, C_t are shared by every channel of the layer
(one group). For channel d = h * P + p of head h the recurrence is the
selective update of Sec. 3 (eq. mamba-scan-background) with

    dt_t[d] = dt_t[h],   A[d, n] = A[h] for every n,   D[d] = D[h],

so the SSD layer is exactly the diagonal layer with tied parameters. Each
function below ties the parameters and then runs the plain fp64 recurrences
of ``oracle/__init__.py`` (the same block restriction, eqs. boundary-state and
partial-reverse of Sec. 4). Nothing is blocked, chunked or reordered here.

Layouts: x [Bt, L, H, P]; dt [Bt, L, H] (after softplus); B, C [Bt, L, N];
A, D [H]; states [Bt, nS, H, P, N] (states[k] follows token (k+1)Bs - 1).

The backward is the diagonal layer's backward with the same tie: a tied
parameter's gradient is the sum of the gradients of the entries it stands for
(dt[h] over the head's channels, A[h] over its channels and state indices,
D[h] over its channels).

Parity status: pinned in ``tests/test_ssd_oracle_pins.py`` by the per-head
semiseparable-matrix form of the block restriction (y = M x with the scalar
decay written as exp of a sum, built independently of any recurrence), the
closed form of the state at a block end, the single-block invariant,
bit-exact caching, and (backward) central finite differences of the pinned
forward for every input, including the tied A, D and dt, plus an exact
matrix-form check of the linear gradients (dx, dB, dC of every stream,
including the clean x and B through the cached states).
"""

from __future__ import annotations

import numpy as np

from . import GRAD_NAMES
from . import active_block as _active_block
from . import backward as _backward
from . import boundary_states as _boundary_states
from . import forward as _forward


def _tie(x, dt, A=None, D=None, N=None):
    """Channel-level tensors of the tied diagonal layer (see the module docstring)."""
    x = np.asarray(x, np.float64)
    Bt, L, H, P = x.shape
    xd = x.reshape(Bt, L, H * P)
    dtd = np.repeat(np.asarray(dt, np.float64), P, axis=2)          # [Bt, L, H*P], d = h*P + p
    Ad = None if A is None else np.repeat(np.asarray(A, np.float64), P)[:, None] * np.ones((1, N))
    Dd = None if D is None else np.repeat(np.asarray(D, np.float64), P)
    return xd, dtd, Ad, Dd


def _heads(a, H, P):
    """[..., H*P] -> [..., H, P]; [Bt, nS, H*P, N] -> [Bt, nS, H, P, N]."""
    if a.ndim == 3:
        return a.reshape(a.shape[0], a.shape[1], H, P)
    return a.reshape(a.shape[0], a.shape[1], H, P, a.shape[3])


def forward(block, x_c, dt_c, B_c, C_c, x_n, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r):
    """All-block forward of the SSD layer. Returns (y_c, y_n, states)."""
    H, P = np.asarray(x_c).shape[2:]
    N = np.asarray(B_c).shape[2]
    xc, dtc, Afd, Dfd = _tie(x_c, dt_c, A_f, D_f, N)
    xn, dtf, _, _ = _tie(x_n, dt_f)
    _, dtr, Ard, Drd = _tie(x_n, dt_r, A_r, D_r, N)
    y_c, y_n, st = _forward(block, xc, dtc, B_c, C_c, xn, dtf, B_f, C_f, dtr, B_r, C_r, Afd, Dfd, Ard, Drd)
    return _heads(y_c, H, P), _heads(y_n, H, P), _heads(st, H, P)


def boundary_states(block, x_c, dt_c, B_c, C_c, A_f, D_f, init_state=None, emit_all=True, want_y=False):
    """Cache build of the SSD layer. Returns (states, y_c or None)."""
    H, P = np.asarray(x_c).shape[2:]
    N = np.asarray(B_c).shape[2]
    xc, dtc, Afd, Dfd = _tie(x_c, dt_c, A_f, D_f, N)
    init = None
    if init_state is not None:
        init = np.asarray(init_state, np.float64).reshape(xc.shape[0], H * P, N)
    st, y = _boundary_states(block, xc, dtc, B_c, C_c, Afd, Dfd, init, emit_all, want_y)
    return _heads(st, H, P), (None if y is None else _heads(y, H, P))


def active_block(seed, x_n, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r):
    """One cached noisy block of the SSD layer (length = block size). Returns y_n."""
    H, P = np.asarray(x_n).shape[2:]
    N = np.asarray(B_f).shape[2]
    xn, dtf, Afd, Dfd = _tie(x_n, dt_f, A_f, D_f, N)
    _, dtr, Ard, Drd = _tie(x_n, dt_r, A_r, D_r, N)
    sd = np.asarray(seed, np.float64).reshape(xn.shape[0], H * P, N)
    y = _active_block(sd, xn, dtf, B_f, C_f, dtr, B_r, C_r, Afd, Dfd, Ard, Drd)
    return _heads(y, H, P)


def backward(block, x_c, dt_c, B_c, C_c, x_n, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r,
             states, dy_c, dy_n, dstates=None):
    """Gradients of <dy_c,y_c> + <dy_n,y_n> + <dstates,states> for the SSD
    layer (states as returned by ``forward``). Returns a dict keyed like the
    inputs, in the SSD layouts; dy_c and dstates may be None."""
    H, P = np.asarray(x_c).shape[2:]
    N = np.asarray(B_c).shape[2]
    xc, dtc, Afd, Dfd = _tie(x_c, dt_c, A_f, D_f, N)
    xn, dtf, _, _ = _tie(x_n, dt_f)
    _, dtr, Ard, Drd = _tie(x_n, dt_r, A_r, D_r, N)
    Bt, L = xc.shape[:2]
    st = np.asarray(states, np.float64).reshape(Bt, -1, H * P, N)
    dyc = None if dy_c is None else np.asarray(dy_c, np.float64).reshape(Bt, L, H * P)
    dyn = np.asarray(dy_n, np.float64).reshape(Bt, L, H * P)
    dst = None if dstates is None else np.asarray(dstates, np.float64).reshape(Bt, -1, H * P, N)
    g = _backward(block, xc, dtc, B_c, C_c, xn, dtf, B_f, C_f, dtr, B_r, C_r, Afd, Dfd, Ard, Drd,
                  st, dyc, dyn, dst)
    out = {}
    for k in GRAD_NAMES:
        a = g[k]
        if k in ("x_c", "x_n"):
            out[k] = a.reshape(Bt, L, H, P)
        elif k in ("dt_c", "dt_f", "dt_r"):
            out[k] = a.reshape(Bt, L, H, P).sum(axis=3)
        elif k in ("A_f", "A_r"):
            out[k] = a.reshape(H, P, N).sum(axis=(1, 2))
        elif k in ("D_f", "D_r"):
            out[k] = a.reshape(H, P).sum(axis=1)
        else:
            out[k] = a
    return out
