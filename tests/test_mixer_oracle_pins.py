"""Pins of the mixer oracle (oracle/mixer.py): convolution, softplus step size
and gated output around the pinned scan oracle.

  * hand-worked convolutions (tap order, initial state, the clean context of
    a noisy block), values written out below;
  * a noisy block equals the clean stream where its inputs equal the clean
    ones, even with different noisy inputs in every other block: its
    convolution reads the clean raw inputs before it (a planted mistake that
    reads the noisy stream there fails);
  * the cache (SSM state and convolution state) reproduces the last noisy
    block bit for bit in fp64, and appending reproduces one scan;
  * central finite differences of every input, the convolution taps, the
    convolution bias and both step-size biases included;
  * identities of softplus and SiLU.
"""

import numpy as np
import pytest

from oracle import mixer


def test_softplus_and_silu_identities():
    z = np.linspace(-30, 30, 601)
    assert np.allclose(mixer.softplus(z) - mixer.softplus(-z), z, rtol=0, atol=1e-12)
    assert np.allclose(mixer.silu(z), z / (1 + np.exp(-z)), rtol=1e-15)
    h = 1e-6
    fd = (mixer.silu(z + h) - mixer.silu(z - h)) / (2 * h)
    assert np.allclose(mixer.dsilu(z), fd, rtol=1e-7, atol=1e-9)


def _one_channel(a):
    return np.asarray(a, np.float64).reshape(1, -1, 1)


def test_hand_worked_convolution():
    # taps w = [1, 10, 100, 1000]: tap 3 multiplies the current token
    w = np.array([[1.0, 10.0, 100.0, 1000.0]])
    z1 = np.zeros(1)
    p = mixer.prep(4, _one_channel([1, 2, 3, 4]), _one_channel([0, 0, 0, 0]), None, None, None, w, z1, z1, z1)
    # 1000*1; 100*1 + 1000*2; 10*1 + 100*2 + 1000*3; 1 + 20 + 300 + 4000
    assert p["pre_c"].ravel().tolist() == [1000.0, 2100.0, 3210.0, 4321.0]
    # initial state [7, 8, 9] (oldest first): token 0 sees 7, 8, 9, 1
    init = np.array([7.0, 8.0, 9.0]).reshape(1, 3, 1)
    p = mixer.prep(4, _one_channel([1, 2, 3, 4]), _one_channel([0, 0, 0, 0]), None, None, None, w, z1, z1, z1, init)
    assert p["pre_c"].ravel()[0] == 7 + 80 + 900 + 1000
    # noisy blocks of 2 tokens: block 1 (tokens 2, 3) reads clean tokens 0, 1
    p = mixer.prep(2, _one_channel([1, 2, 3, 4]), _one_channel([0] * 4), _one_channel([5, 6, 7, 8]),
                   _one_channel([0] * 4), _one_channel([0] * 4), w, z1, z1, z1)
    # 1000*5; 100*5 + 1000*6; 10*1 + 100*2 + 1000*7; 1*1 + 10*2 + 100*7 + 1000*8
    assert p["pre_n"].ravel().tolist() == [5000.0, 6500.0, 7210.0, 8721.0]


def _problem(Bt=2, L=12, Bs=4, D=3, N=4, seed=0):
    r = np.random.default_rng(seed)
    td = lambda: r.normal(size=(Bt, L, D))
    tn = lambda: r.normal(size=(Bt, L, N)) / 2
    d = {"xr_c": td(), "dtr_c": r.normal(-2, 0.5, size=(Bt, L, D)), "B_c": tn(), "C_c": tn(), "z_c": td(),
         "xr_n": td(), "dtr_f": r.normal(-2, 0.5, size=(Bt, L, D)), "B_f": tn(), "C_f": tn(),
         "dtr_r": r.normal(-2, 0.5, size=(Bt, L, D)), "B_r": tn(), "C_r": tn(), "z_n": td(),
         "A_f": -np.exp(r.uniform(0, np.log(16), size=(D, N))), "D_f": r.normal(0, 0.1, size=D),
         "A_r": -np.exp(r.uniform(0, np.log(16), size=(D, N))), "D_r": r.normal(0, 0.1, size=D),
         "w": r.normal(0, 0.5, size=(D, 4)), "b": r.normal(0, 0.1, size=D),
         "bias_f": r.normal(0, 0.3, size=D), "bias_r": r.normal(0, 0.3, size=D)}
    return d


FWD = ("xr_c", "dtr_c", "B_c", "C_c", "z_c", "xr_n", "dtr_f", "B_f", "C_f", "dtr_r", "B_r", "C_r", "z_n",
       "A_f", "D_f", "A_r", "D_r", "w", "b", "bias_f", "bias_r")


def test_noisy_convolution_reads_the_clean_context():
    Bs = 4
    d = _problem(L=16, Bs=Bs, seed=1)
    for k in range(4):
        q = dict(d)
        sl = slice(k * Bs, (k + 1) * Bs)
        # noisy inputs equal the clean ones in block k, differ everywhere else
        for a, c in (("xr_n", "xr_c"), ("dtr_f", "dtr_c"), ("B_f", "B_c"), ("C_f", "C_c"), ("z_n", "z_c")):
            q[a] = q[a].copy()
            q[a][:, sl] = q[c][:, sl]
        q["B_r"] = np.zeros_like(q["B_r"])
        q["D_r"] = np.zeros_like(q["D_r"])
        oc, on, _ = mixer.forward(Bs, *[q[n] for n in FWD])
        assert np.array_equal(on[:, sl], oc[:, sl]), k


def test_planted_mistake_noisy_context_breaks_the_invariant():
    """A convolution that reads the noisy stream before the block (instead of
    the clean one) fails the invariant above."""
    Bs = 4
    d = _problem(L=16, Bs=Bs, seed=2)
    k = 2
    sl = slice(k * Bs, (k + 1) * Bs)
    q = dict(d)
    for a, c in (("xr_n", "xr_c"), ("dtr_f", "dtr_c"), ("B_f", "B_c"), ("C_f", "C_c"), ("z_n", "z_c")):
        q[a] = q[a].copy()
        q[a][:, sl] = q[c][:, sl]
    q["B_r"] = np.zeros_like(q["B_r"])
    q["D_r"] = np.zeros_like(q["D_r"])
    orig = mixer._windows

    def wrong(xr_c, xr_n, block, conv_init):
        wc, _ = orig(xr_c, None, block, conv_init)
        wn, _ = orig(xr_n, None, block, conv_init)  # noisy stream throughout
        return wc, wn

    try:
        mixer._windows = wrong
        oc, on, _ = mixer.forward(Bs, *[q[n] for n in FWD])
    finally:
        mixer._windows = orig
    assert not np.allclose(on[:, sl], oc[:, sl], rtol=1e-6, atol=1e-9)


@pytest.mark.parametrize("Bs", [1, 2, 4])
def test_cache_with_convolution_state_is_exact(Bs):
    L = 4 * max(Bs, 2)
    d = _problem(L=L, Bs=Bs, seed=3)
    oc, on, st = mixer.forward(Bs, *[d[n] for n in FWD])
    pre = {k: (v[:, : L - Bs] if np.ndim(v) == 3 else v) for k, v in d.items()}
    s, cs = mixer.boundary_states(Bs, pre["xr_c"], pre["dtr_c"], pre["B_c"], pre["C_c"], d["A_f"], d["D_f"],
                                  d["w"], d["b"], d["bias_f"], emit_all=True)
    assert np.array_equal(s, st[:, :-1])
    blk = {k: (v[:, L - Bs:] if np.ndim(v) == 3 else v) for k, v in d.items()}
    y = mixer.active_block(s[:, -1], cs[:, -1], blk["xr_n"], blk["dtr_f"], blk["B_f"], blk["C_f"], blk["dtr_r"],
                           blk["B_r"], blk["C_r"], blk["z_n"], d["A_f"], d["D_f"], d["A_r"], d["D_r"], d["w"],
                           d["b"], d["bias_f"], d["bias_r"])
    assert np.array_equal(y, on[:, L - Bs:])


def test_cache_append_matches_one_scan():
    Bs, L = 4, 16
    d = _problem(L=L, Bs=Bs, seed=4)
    args = ("dtr_c", "B_c", "C_c")
    full_s, full_c = mixer.boundary_states(Bs, d["xr_c"], *[d[k] for k in args], d["A_f"], d["D_f"], d["w"], d["b"],
                                           d["bias_f"], emit_all=False)
    h = 8
    a_s, a_c = mixer.boundary_states(Bs, d["xr_c"][:, :h], *[d[k][:, :h] for k in args], d["A_f"], d["D_f"],
                                     d["w"], d["b"], d["bias_f"], emit_all=False)
    b_s, b_c = mixer.boundary_states(Bs, d["xr_c"][:, h:], *[d[k][:, h:] for k in args], d["A_f"], d["D_f"],
                                     d["w"], d["b"], d["bias_f"], init_state=a_s[:, 0], conv_init=a_c[:, 0],
                                     emit_all=False)
    assert np.allclose(b_s, full_s, rtol=1e-12, atol=1e-14)
    assert np.array_equal(b_c, full_c)


def test_finite_differences_of_every_input():
    Bs = 4
    d = _problem(L=12, Bs=Bs, seed=5)
    r = np.random.default_rng(6)
    dout_c = r.normal(size=d["xr_c"].shape)
    dout_n = r.normal(size=d["xr_c"].shape)
    dst = r.normal(size=(2, 3, 3, 4))
    g = mixer.backward(Bs, *[d[n] for n in FWD], dout_c, dout_n, dst)

    def loss(q):
        oc, on, st = mixer.forward(Bs, *[q[n] for n in FWD])
        return np.sum(dout_c * oc) + np.sum(dout_n * on) + np.sum(dst * st)

    h = 1e-6
    for name in FWD:
        v = r.normal(size=np.shape(d[name]))
        qp, qm = dict(d), dict(d)
        qp[name] = d[name] + h * v
        qm[name] = d[name] - h * v
        fd = (loss(qp) - loss(qm)) / (2 * h)
        an = float(np.sum(g[name] * v))
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (name, fd, an)
