"""Pins of the SSD (Mamba-2 form) oracle, CPU only.

The oracle ties the diagonal layer's parameters per head (Appendix C's Mamba-2
mixers: one decay per head, B and C shared by all channels). Here the block
restriction of Sec. 4 (eqs. boundary-state and partial-reverse) is written
out per head as the explicit semiseparable matrix of the SSD form: decays are
exp(A * sum of dt) summed directly over index ranges, so no recurrence and no
channel/head flattening is shared with the oracle. A wrong head/channel map,
a decay index off by one, a dropped reverse or seed term or a wrong D sum
each fails here.
"""

import numpy as np
import pytest

from oracle import ssd


def _inputs(seed, Bt=2, L=12, Bs=4, H=2, P=3, N=4):
    rng = np.random.default_rng(seed)
    sp = lambda z: np.log1p(np.exp(z))
    g = lambda *s: rng.standard_normal(s)
    d = dict(x_c=g(Bt, L, H, P), dt_c=sp(rng.normal(-1, .5, (Bt, L, H))), B_c=g(Bt, L, N), C_c=g(Bt, L, N),
             x_n=g(Bt, L, H, P), dt_f=sp(rng.normal(-1, .5, (Bt, L, H))), B_f=g(Bt, L, N), C_f=g(Bt, L, N),
             dt_r=sp(rng.normal(-1, .5, (Bt, L, H))), B_r=g(Bt, L, N), C_r=g(Bt, L, N),
             A_f=-np.exp(rng.uniform(0, np.log(4), H)), D_f=rng.normal(0, .3, H),
             A_r=-np.exp(rng.uniform(0, np.log(4), H)), D_r=rng.normal(0, .3, H))
    return Bs, d


NAMES = ("x_c", "dt_c", "B_c", "C_c", "x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r", "A_f", "D_f", "A_r", "D_r")


def _dsum(dt, lo, hi):
    """sum of dt[r] for lo <= r <= hi (0 if the range is empty), by a plain loop."""
    s = 0.0
    for r in range(lo, hi + 1):
        s += dt[r]
    return s


def matrix_form(Bs, d):
    """Per batch row and head: clean output, block-end states, noisy output."""
    Bt, L, H, P = d["x_c"].shape
    N = d["B_c"].shape[2]
    nb = L // Bs
    y_c = np.zeros((Bt, L, H, P))
    y_n = np.zeros((Bt, L, H, P))
    st = np.zeros((Bt, nb, H, P, N))
    for b in range(Bt):
        for h in range(H):
            dc, df, dr = d["dt_c"][b, :, h], d["dt_f"][b, :, h], d["dt_r"][b, :, h]
            Af, Ar = d["A_f"][h], d["A_r"][h]
            xc, xn = d["x_c"][b, :, h, :], d["x_n"][b, :, h, :]
            # clean: lower-triangular semiseparable matrix over the whole stream
            Mc = np.zeros((L, L))
            for t in range(L):
                for s in range(t + 1):
                    Mc[t, s] = d["C_c"][b, t] @ d["B_c"][b, s] * np.exp(Af * _dsum(dc, s + 1, t)) * dc[s]
            y_c[b, :, h, :] = Mc @ xc + d["D_f"][h] * xc
            # block-end states: sum over all earlier tokens of decay * dt * x B^T
            for k in range(nb):
                e = (k + 1) * Bs - 1
                for s in range(e + 1):
                    st[b, k, h] += np.exp(Af * _dsum(dc, s + 1, e)) * dc[s] * np.outer(xc[s], d["B_c"][b, s])
            # noisy blocks: seeded forward (lower) + block-local reverse (upper)
            for k in range(nb):
                lo, hi = k * Bs, (k + 1) * Bs - 1
                seed = st[b, k - 1, h] if k > 0 else np.zeros((P, N))
                for t in range(lo, hi + 1):
                    acc = d["C_f"][b, t] @ (np.exp(Af * _dsum(df, lo, t)) * seed).T
                    for s in range(lo, t + 1):
                        acc = acc + (d["C_f"][b, t] @ d["B_f"][b, s]) * np.exp(Af * _dsum(df, s + 1, t)) * df[s] * xn[s]
                    for s in range(t, hi + 1):
                        acc = acc + (d["C_r"][b, t] @ d["B_r"][b, s]) * np.exp(Ar * _dsum(dr, t, s - 1)) * dr[s] * xn[s]
                    y_n[b, t, h] = acc + (d["D_f"][h] + d["D_r"][h]) * xn[t]
    return y_c, y_n, st


@pytest.mark.parametrize("seed,Bs", [(0, 4), (1, 1), (2, 12), (3, 3)])
def test_ssd_forward_matches_matrix_form(seed, Bs):
    _, d = _inputs(seed, Bs=Bs)
    y_c, y_n, st = ssd.forward(Bs, *[d[k] for k in NAMES])
    m_c, m_n, m_st = matrix_form(Bs, d)
    for got, want in ((y_c, m_c), (y_n, m_n), (st, m_st)):
        assert np.max(np.abs(got - want)) <= 1e-11 * max(1.0, np.max(np.abs(want)))


def test_ssd_cache_exactness_and_single_block():
    Bs, d = _inputs(4, L=12, Bs=4)
    y_c, y_n, st = ssd.forward(Bs, *[d[k] for k in NAMES])
    # cache build alone gives the same states bit for bit; every noisy block
    # recomputed from its cached seed equals the all-block output bit for bit
    st2, y2 = ssd.boundary_states(Bs, d["x_c"], d["dt_c"], d["B_c"], d["C_c"], d["A_f"], d["D_f"], want_y=True)
    assert np.array_equal(st, st2) and np.array_equal(y_c, y2)
    for k in range(12 // Bs):
        sl = slice(k * Bs, (k + 1) * Bs)
        seed = st[:, k - 1] if k > 0 else np.zeros_like(st[:, 0])
        ya = ssd.active_block(seed, d["x_n"][:, sl], d["dt_f"][:, sl], d["B_f"][:, sl], d["C_f"][:, sl],
                              d["dt_r"][:, sl], d["B_r"][:, sl], d["C_r"][:, sl],
                              d["A_f"], d["D_f"], d["A_r"], d["D_r"])
        assert np.array_equal(ya, y_n[:, sl])
    # cache append: states of the second half from the first half's last state
    st_a, _ = ssd.boundary_states(Bs, *[d[k][:, :8] for k in ("x_c", "dt_c", "B_c", "C_c")], d["A_f"], d["D_f"])
    st_b, _ = ssd.boundary_states(Bs, *[d[k][:, 8:] for k in ("x_c", "dt_c", "B_c", "C_c")], d["A_f"], d["D_f"],
                                  init_state=st_a[:, -1])
    assert np.array_equal(st_b[:, -1], st[:, -1])


def test_ssd_planted_head_map_fails(monkeypatch):
    """A planted channel-major tie (d = p*H + h instead of h*P + p) in the oracle
    is caught by the matrix form."""
    Bs, d = _inputs(5)
    m_c, m_n, _ = matrix_form(Bs, d)

    def bad_tie(x, dt, A=None, D=None, N=None):
        x = np.asarray(x, np.float64)
        Bt, L, H, P = x.shape
        xd = x.reshape(Bt, L, H * P)
        dtd = np.tile(np.asarray(dt, np.float64), (1, 1, P))
        Ad = None if A is None else np.tile(np.asarray(A, np.float64), P)[:, None] * np.ones((1, N))
        Dd = None if D is None else np.tile(np.asarray(D, np.float64), P)
        return xd, dtd, Ad, Dd

    monkeypatch.setattr(ssd, "_tie", bad_tie)
    y_c, y_n, _ = ssd.forward(Bs, *[d[k] for k in NAMES])
    assert np.max(np.abs(y_c - m_c)) > 1e-3 and np.max(np.abs(y_n - m_n)) > 1e-3


@pytest.mark.parametrize("seed,Bs", [(0, 4), (6, 3)])
def test_ssd_backward_matches_finite_differences(seed, Bs):
    """Central differences of the pinned SSD forward, along a random direction
    per input, against the oracle's gradients of <dy_c,y_c>+<dy_n,y_n>+<dS,S>
    (tied A, D and dt included)."""
    _, d = _inputs(seed, Bs=Bs)
    y_c, y_n, st = ssd.forward(Bs, *[d[k] for k in NAMES])
    rng = np.random.default_rng(100 + seed)
    dyc, dyn, dst = rng.standard_normal(y_c.shape), rng.standard_normal(y_n.shape), rng.standard_normal(st.shape)
    g = ssd.backward(Bs, *[d[k] for k in NAMES], st, dyc, dyn, dst)

    def loss(dd):
        a, b, c = ssd.forward(Bs, *[dd[k] for k in NAMES])
        return float((a * dyc).sum() + (b * dyn).sum() + (c * dst).sum())

    for k in NAMES:
        v = rng.standard_normal(d[k].shape)
        eps = 1e-6
        dp, dm = dict(d), dict(d)
        dp[k], dm[k] = d[k] + eps * v, d[k] - eps * v
        fd = (loss(dp) - loss(dm)) / (2 * eps)
        an = float((g[k] * v).sum())
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (k, an, fd)


def _kernel(dt, A, lo, hi, t, s):
    """decay * dt_s of the forward (s <= t) direction inside [lo, hi]."""
    return np.exp(A * _dsum(dt, s + 1, t)) * dt[s]


def test_ssd_backward_linear_gradients_matrix_form():
    """dx, dB and dC of the oracle's SSD backward against the same gradients
    written out from the semiseparable matrix form (explicit sums; the clean
    x and B also receive the gradient through the cached block-end states, as
    the seed of every next noisy block and through dstates)."""
    Bs, d = _inputs(7, Bt=1, L=8, Bs=4, H=2, P=2, N=3)
    Bt, L, H, P = d["x_c"].shape
    N = d["B_c"].shape[2]
    nb = L // Bs
    y_c, y_n, st = ssd.forward(Bs, *[d[k] for k in NAMES])
    rng = np.random.default_rng(11)
    dyc, dyn, dst = rng.standard_normal(y_c.shape), rng.standard_normal(y_n.shape), rng.standard_normal(st.shape)
    g = ssd.backward(Bs, *[d[k] for k in NAMES], st, dyc, dyn, dst)
    b = 0
    want = {k: np.zeros_like(d[k]) for k in ("x_c", "x_n", "B_c", "C_c", "B_f", "C_f", "B_r", "C_r")}
    for h in range(H):
        dc, df, dr = d["dt_c"][b, :, h], d["dt_f"][b, :, h], d["dt_r"][b, :, h]
        Af, Ar, Df, Dr = d["A_f"][h], d["A_r"][h], d["D_f"][h], d["D_r"][h]
        xc, xn = d["x_c"][b, :, h], d["x_n"][b, :, h]
        Bc, Cc, Bf, Cf, Br, Cr = (d[k][b] for k in ("B_c", "C_c", "B_f", "C_f", "B_r", "C_r"))
        # total gradient of each block-end state: dstates + the seed term of the next noisy block
        Gk = np.array(dst[b, :, h], dtype=float)
        for k in range(nb - 1):
            lo, hi = (k + 1) * Bs, (k + 2) * Bs - 1
            for t in range(lo, hi + 1):
                Gk[k] += np.exp(Af * _dsum(df, lo, t)) * np.outer(dyn[b, t, h], Cf[t])
        # clean stream: y_c = sum_s (C_t . B_s) K_ts x_s + D_f x_t over the whole stream
        for t in range(L):
            want["x_c"][b, t, h] += Df * dyc[b, t, h]
            for s in range(t + 1):
                K = _kernel(dc, Af, 0, L - 1, t, s)
                gts = Cc[t] @ Bc[s]
                want["x_c"][b, s, h] += gts * K * dyc[b, t, h]
                q = dyc[b, t, h] @ xc[s]
                want["C_c"][b, t] += q * K * Bc[s]
                want["B_c"][b, s] += q * K * Cc[t]
        # clean x and B through the states: S_k = sum_{s <= e_k} exp(A sum_{s<r<=e_k} dt) dt_s x_s B_s^T
        for k in range(nb):
            e = (k + 1) * Bs - 1
            for s in range(e + 1):
                w = _kernel(dc, Af, 0, e, e, s)
                want["x_c"][b, s, h] += w * (Gk[k] @ Bc[s])
                want["B_c"][b, s] += w * (xc[s] @ Gk[k])
        # noisy blocks: forward (lower, with seed), reverse (upper), D terms
        for k in range(nb):
            lo, hi = k * Bs, (k + 1) * Bs - 1
            seed = st[b, k - 1, h] if k > 0 else np.zeros((P, N))
            for t in range(lo, hi + 1):
                want["x_n"][b, t, h] += (Df + Dr) * dyn[b, t, h]
                want["C_f"][b, t] += np.exp(Af * _dsum(df, lo, t)) * (dyn[b, t, h] @ seed)
                for s in range(lo, t + 1):
                    K = _kernel(df, Af, lo, hi, t, s)
                    q = dyn[b, t, h] @ xn[s]
                    want["x_n"][b, s, h] += (Cf[t] @ Bf[s]) * K * dyn[b, t, h]
                    want["C_f"][b, t] += q * K * Bf[s]
                    want["B_f"][b, s] += q * K * Cf[t]
                for s in range(t, hi + 1):
                    K = np.exp(Ar * _dsum(dr, t, s - 1)) * dr[s]
                    q = dyn[b, t, h] @ xn[s]
                    want["x_n"][b, s, h] += (Cr[t] @ Br[s]) * K * dyn[b, t, h]
                    want["C_r"][b, t] += q * K * Br[s]
                    want["B_r"][b, s] += q * K * Cr[t]
    for k, v in want.items():
        assert np.max(np.abs(g[k] - v)) <= 1e-11 * max(1.0, np.max(np.abs(v))), k
