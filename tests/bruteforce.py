"""Explicit semiseparable-matrix form of the block-restricted bidirectional scan.

Test helper, independent of the oracle's recurrences: every output is written
as a sum over source positions s of a decay factor exp(A * sum of dt over the
positions between s and t) times the input at s, with the sums of dt formed
explicitly for each (t, s) pair. Nothing here runs a recurrence, so an error
in the oracle's step order, indexing or seeding shows up as a mismatch.

For the selective update of Sec. 3 with a_t = exp(dt_t A):
  forward scan:  h_t = sum_{s<=t} exp(A sum_{r=s+1..t} dt_r) dt_s B_s x_s
  reverse scan:  h_t = sum_{s>=t} exp(A sum_{r=t..s-1} dt_r) dt_s B_s x_s
  seeded block:  h_t += exp(A sum_{r=t0..t} dt_r) seed
Sizes must be tiny (O(L^2 D N) work with Python-level loops over t, s).
"""

from __future__ import annotations

import numpy as np


def _fwd_state(dt, B, x, A, t, s_lo):
    """sum_{s=s_lo..t} exp(A * sum_{r=s+1..t} dt_r) dt_s B_s x_s for one channel.
    dt, x: [L]; B: [L, N]; A: [N]."""
    out = np.zeros(A.shape[0])
    for s in range(s_lo, t + 1):
        tot = 0.0
        for r in range(s + 1, t + 1):
            tot += dt[r]
        out += np.exp(A * tot) * dt[s] * B[s] * x[s]
    return out


def _rev_state(dt, B, x, A, t, s_hi):
    out = np.zeros(A.shape[0])
    for s in range(t, s_hi + 1):
        tot = 0.0
        for r in range(t, s):
            tot += dt[r]
        out += np.exp(A * tot) * dt[s] * B[s] * x[s]
    return out


def _seed_decay(dt, A, t0, t):
    tot = 0.0
    for r in range(t0, t + 1):
        tot += dt[r]
    return np.exp(A * tot)


def forward(block, w):
    """Brute-force all-block forward. w: dict of fp64 arrays (inputs.py names).
    Returns (y_c, y_n, states)."""
    x_c, dt_c, B_c, C_c = w["x_c"], w["dt_c"], w["B_c"], w["C_c"]
    x_n = w["x_n"]
    Bt, L, D = x_c.shape
    N = B_c.shape[2]
    nb = L // block
    y_c = np.zeros((Bt, L, D))
    y_n = np.zeros((Bt, L, D))
    st = np.zeros((Bt, nb, D, N))
    for b in range(Bt):
        for d in range(D):
            Af, Ar = w["A_f"][d], w["A_r"][d]
            Df, Dr = w["D_f"][d], w["D_r"][d]
            for t in range(L):
                h = _fwd_state(dt_c[b, :, d], B_c[b], x_c[b, :, d], Af, t, 0)
                y_c[b, t, d] = C_c[b, t] @ h + Df * x_c[b, t, d]
            for k in range(nb):
                st[b, k, d] = _fwd_state(dt_c[b, :, d], B_c[b], x_c[b, :, d], Af, (k + 1) * block - 1, 0)
            for k in range(nb):
                t0, t1 = k * block, (k + 1) * block - 1
                seed = st[b, k - 1, d] if k > 0 else np.zeros(N)
                for t in range(t0, t1 + 1):
                    hf = _fwd_state(w["dt_f"][b, :, d], w["B_f"][b], x_n[b, :, d], Af, t, t0)
                    hf = hf + _seed_decay(w["dt_f"][b, :, d], Af, t0, t) * seed
                    hr = _rev_state(w["dt_r"][b, :, d], w["B_r"][b], x_n[b, :, d], Ar, t, t1)
                    y_n[b, t, d] = (w["C_f"][b, t] @ hf + Df * x_n[b, t, d]
                                    + w["C_r"][b, t] @ hr + Dr * x_n[b, t, d])
    return y_c, y_n, st


def linear_map_x(block, w):
    """The matrix J with (y_c, y_n, states) = J (x_c, x_n), built column by
    column from the brute-force forward (the outputs are linear in x)."""
    Bt, L, D = w["x_c"].shape
    nx = Bt * L * D
    cols = []
    base = dict(w)
    for which in ("x_c", "x_n"):
        for i in range(nx):
            e = np.zeros(nx)
            e[i] = 1.0
            ww = dict(base)
            ww["x_c"] = np.zeros((Bt, L, D))
            ww["x_n"] = np.zeros((Bt, L, D))
            ww[which] = e.reshape(Bt, L, D)
            y_c, y_n, st = forward(block, ww)
            cols.append(np.concatenate([y_c.ravel(), y_n.ravel(), st.ravel()]))
    return np.stack(cols, axis=1)
