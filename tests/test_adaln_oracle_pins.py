"""Pins of the AdaLN active-block oracle (oracle/adaln.py) against facts fixed
by the definition of layer norm and of the gated residual, independent of how
the oracle computes them (Appendix E, eq. cacheable-adaln):

  * LN output per token has mean 0 and variance var / (var + eps) (closed form);
  * scale = -1 removes the normalised input: u equals the shift, whatever h is;
  * the step's mixer part is invariant to any per-token affine map of h,
    h -> a_t h + b_t with a_t > 0 (eps = 0): a wrong reduction axis, a missing
    centring or a missing division breaks it (a planted mistake shows this);
  * gate = 0 returns h exactly; the cached seed is never modified.
"""

import numpy as np
import pytest

from oracle import adaln


def _problem(Bt=2, Bs=8, D=24, N=4, seed=0):
    r = np.random.default_rng(seed)
    d = {
        "seed": r.normal(size=(Bt, D, N)),
        "h": r.normal(1.5, 2.0, size=(Bt, Bs, D)),
        "dt_f": np.log1p(np.exp(r.normal(-2, 0.5, size=(Bt, Bs, D)))),
        "dt_r": np.log1p(np.exp(r.normal(-2, 0.5, size=(Bt, Bs, D)))),
        "B_f": r.normal(size=(Bt, Bs, N)) / 2, "C_f": r.normal(size=(Bt, Bs, N)) / 2,
        "B_r": r.normal(size=(Bt, Bs, N)) / 2, "C_r": r.normal(size=(Bt, Bs, N)) / 2,
        "A_f": -np.exp(r.uniform(0, np.log(16), size=(D, N))), "A_r": -np.exp(r.uniform(0, np.log(16), size=(D, N))),
        "D_f": r.normal(0, 0.1, size=D), "D_r": r.normal(0, 0.1, size=D),
        "shift": r.normal(0, 0.3, size=(Bt, D)), "scale": r.normal(0, 0.3, size=(Bt, D)),
        "gate": r.normal(1, 0.3, size=(Bt, D)),
    }
    return d


def _run(d, h=None, eps=1e-5, **over):
    q = dict(d)
    q.update(over)
    return adaln.active_block_adaln(q["seed"], d["h"] if h is None else h, q["dt_f"], q["B_f"], q["C_f"], q["dt_r"],
                                    q["B_r"], q["C_r"], q["A_f"], q["D_f"], q["A_r"], q["D_r"], q["shift"],
                                    q["scale"], q["gate"], eps)


@pytest.mark.parametrize("eps", [0.0, 1e-5, 0.3])
def test_layer_norm_moments(eps):
    h = np.random.default_rng(1).normal(3.0, 5.0, size=(3, 7, 40))
    z = adaln.layer_norm(h, eps)
    var = h.var(axis=-1)
    assert np.max(np.abs(z.mean(axis=-1))) < 1e-12
    assert np.allclose((z * z).mean(axis=-1), var / (var + eps), rtol=1e-12, atol=0)


def test_scale_minus_one_leaves_only_the_shift():
    d = _problem()
    u = adaln.modulate(d["h"], d["shift"], -np.ones_like(d["scale"]), 1e-5)
    assert np.array_equal(u, np.broadcast_to(d["shift"][:, None, :], u.shape))


def test_gate_zero_returns_h_exactly():
    d = _problem(seed=2)
    out = _run(d, gate=np.zeros_like(d["gate"]))
    assert np.array_equal(out, d["h"])


def test_mixer_part_is_invariant_to_per_token_affine_maps():
    d = _problem(seed=3)
    r = np.random.default_rng(4)
    a = np.exp(r.normal(0, 1, size=d["h"].shape[:2] + (1,)))
    b = r.normal(0, 3, size=d["h"].shape[:2] + (1,))
    h2 = a * d["h"] + b
    m1 = _run(d, eps=0.0) - d["h"]
    m2 = _run(d, h=h2, eps=0.0) - h2
    assert np.max(np.abs(m1 - m2)) <= 1e-10 * np.max(np.abs(m1))


def test_planted_mistake_normalising_over_tokens_breaks_the_invariance():
    """The same invariance computed with LN taken over the token axis (a
    plausible transposition mistake) fails, so the pin above catches it."""
    d = _problem(seed=5)

    def wrong_ln(h, eps):
        h = np.asarray(h, np.float64)
        mu = h.mean(axis=1, keepdims=True)
        var = ((h - mu) ** 2).mean(axis=1, keepdims=True)
        return (h - mu) / np.sqrt(var + eps)

    r = np.random.default_rng(6)
    a = np.exp(r.normal(0, 1, size=d["h"].shape[:2] + (1,)))
    b = r.normal(0, 3, size=d["h"].shape[:2] + (1,))
    h2 = a * d["h"] + b
    orig = adaln.layer_norm
    try:
        adaln.layer_norm = wrong_ln
        m1 = _run(d, eps=0.0) - d["h"]
        m2 = _run(d, h=h2, eps=0.0) - h2
    finally:
        adaln.layer_norm = orig
    assert np.max(np.abs(m1 - m2)) > 1e-3 * np.max(np.abs(m1))


def test_cached_seed_is_read_only():
    d = _problem(seed=7)
    before = d["seed"].copy()
    for step in range(3):
        _run(d, shift=d["shift"] * step, scale=d["scale"] * step)
    assert np.array_equal(before, d["seed"])
