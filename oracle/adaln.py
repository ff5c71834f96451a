"""fp64 oracle of the timestep-modulated active block (adaptive layer norm on
the active block only), for the AdaLN factorization of the paper (Appendix E,
eq. cacheable-adaln).

TEST INFRASTRUCTURE, like the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and the CPU baseline of ``bench.py`` may use it.

The paper maps the timestep embedding e_t to shift, scale and gate vectors and
modulates a layer-normalised hidden state with them,
    u = (1 + scale) * LN(h) + shift,
before the mixer, with the gate applied to the mixer's output on the residual
path. A cacheable layer applies this only to the active block: the clean
prefix path, and therefore the cached boundary state, carries no timestep.

Readings (the paper gives the form, not every detail):
  * LN normalises each token over the channel axis, with the biased variance
    and eps inside the square root, and has no learned affine of its own (the
    modulation plays that role).
  * The in/out projections of the mixer are outside the scan; the modulation
    acts in the scan's channel space, on the noisy block's input x. The
    block's dt, B and C are given (they are projections the caller makes).
  * The residual output of the step is h + gate * y_n, with y_n the
    block-restricted bidirectional output of the modulated input (both
    directions and both skip terms, as in ``active_block``).

Steps, in the paper's order: LN of h, modulation (``modulate``), the cached
active-block scan of the pinned diagonal oracle on u (``active_block``), then
the gated residual. Pins: tests/test_adaln_oracle_pins.py.
"""

from __future__ import annotations

import numpy as np

from . import active_block as _active_block


def layer_norm(h, eps):
    """LN over the last (channel) axis: (h - mean) / sqrt(var + eps)."""
    h = np.asarray(h, np.float64)
    mu = h.mean(axis=-1, keepdims=True)
    var = ((h - mu) ** 2).mean(axis=-1, keepdims=True)
    return (h - mu) / np.sqrt(var + eps)


def modulate(h, shift, scale, eps):
    """u = (1 + scale) * LN(h) + shift. h [Bt, Bs, D]; shift, scale [Bt, D]."""
    shift = np.asarray(shift, np.float64)[:, None, :]
    scale = np.asarray(scale, np.float64)[:, None, :]
    return (1.0 + scale) * layer_norm(h, eps) + shift


def active_block_adaln(seed, h, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r, shift, scale, gate, eps):
    """One timestep-modulated active-block step from the read-only cached seed.
    Returns h + gate * y_n [Bt, Bs, D]."""
    h = np.asarray(h, np.float64)
    u = modulate(h, shift, scale, eps)
    y = _active_block(seed, u, dt_f, B_f, C_f, dt_r, B_r, C_r, A_f, D_f, A_r, D_r)
    return h + np.asarray(gate, np.float64)[:, None, :] * y
