"""CPU check of the decomposition the SSD-form backward kernels follow (fp64
numpy, small sizes): per block and head, the products Q = dy x^T and
G = C B^T, the masked decays M' = G o decay, D = M'^T dy (dx = diag(dt) D,
and the column sums of R' = Q o M' as x_s . D_s), row and column sums turned
into dt and A gradients by a cumulative sum inside the block, the seed terms,
a reverse pass over block-end states, and the transpose of the block-state
product. Its gradients must equal the oracle's (tied diagonal backward) for
every input.
Everything here is written from the matrix form of Sec. 4 (eqs.
boundary-state and partial-reverse) with scalar decays per head."""

import numpy as np
import pytest

from oracle import ssd
from test_ssd_oracle_pins import NAMES, _inputs


def _direction(dy, x, dt, B, C, A, seed, upper):
    """Gradients of <dy, y> for one direction of one block and head:
    y = (mask o (C B^T) o decay) diag(dt) x + diag(E) C seed^T (seed only for
    the forward direction). Returns dx, dB, dC, ddt, dA, dseed."""
    T = len(dt)
    c = np.cumsum(dt[::-1])[::-1] if upper else np.cumsum(dt)  # inclusive suffix / prefix sums
    diff = c[:, None] - c[None, :]                             # c_t - c_s
    mask = np.triu(np.ones((T, T))) if upper else np.tril(np.ones((T, T)))
    dec = np.exp(A * np.where(mask > 0, diff, 0.0)) * mask
    G = C @ B.T
    Mp = G * dec                                               # M' (without dt_s)
    Q = dy @ x.T                                               # dy_t . x_s
    R = Q * Mp * dt[None, :]                                   # R = R' diag(dt), R' = Q o M'
    dG = Q * dec * dt[None, :]
    D = Mp.T @ dy                                              # D_s = sum_t M'[t, s] dy_t
    dx = dt[:, None] * D
    colsum = np.sum(x * D, axis=1)                             # colsum_s R' = x_s . D_s
    dC = dG @ B
    dB = dG.T @ C
    rowdot = np.zeros(T)
    dseed = np.zeros_like(seed) if seed is not None else None
    if seed is not None:
        E = np.exp(A * c)
        Ys = (C @ seed.T) * E[:, None]                         # the seed term of y
        rowdot = np.sum(dy * Ys, axis=1)                       # dy_t . seed term_t
        dC = dC + E[:, None] * (dy @ seed)
        dseed = (E[:, None] * dy).T @ C
    dc = A * (R.sum(axis=1) - dt * colsum + rowdot)
    # c_t = sum of dt over q <= t (forward) or q >= t (reverse)
    ddt = colsum + (np.cumsum(dc[::-1])[::-1] if not upper else np.cumsum(dc))
    dA = float(np.sum(c * dc)) / A
    return dx, dB, dC, ddt, dA, dseed


def planned_backward(Bs, d, states, dyc, dyn, dst):
    Bt, L, H, P = d["x_c"].shape
    N = d["B_c"].shape[2]
    nb = L // Bs
    g = {k: np.zeros_like(d[k]) for k in NAMES}
    for b in range(Bt):
        for h in range(H):
            Af, Ar, Df, Dr = d["A_f"][h], d["A_r"][h], d["D_f"][h], d["D_r"][h]
            gseed = np.zeros((nb, P, N))  # gradient of states[k] through block k+1's seeds
            for k in range(nb):
                sl = slice(k * Bs, (k + 1) * Bs)
                seed = states[b, k - 1, h] if k > 0 else np.zeros((P, N))
                xn = d["x_n"][b, sl, h]
                # noisy block: forward direction (seeded) + block-local reverse
                fx, fB, fC, fdt, fA, fS = _direction(dyn[b, sl, h], xn, d["dt_f"][b, sl, h], d["B_f"][b, sl],
                                                     d["C_f"][b, sl], Af, seed, False)
                rx, rB, rC, rdt, rA, _ = _direction(dyn[b, sl, h], xn, d["dt_r"][b, sl, h], d["B_r"][b, sl],
                                                    d["C_r"][b, sl], Ar, None, True)
                g["x_n"][b, sl, h] += fx + rx + (Df + Dr) * dyn[b, sl, h]
                g["B_f"][b, sl] += fB
                g["C_f"][b, sl] += fC
                g["B_r"][b, sl] += rB
                g["C_r"][b, sl] += rC
                g["dt_f"][b, sl, h] += fdt
                g["dt_r"][b, sl, h] += rdt
                g["A_f"][h] += fA
                g["A_r"][h] += rA
                g["D_f"][h] += np.sum(dyn[b, sl, h] * xn)
                g["D_r"][h] += np.sum(dyn[b, sl, h] * xn)
                # clean block: forward direction seeded with the state before it
                xc = d["x_c"][b, sl, h]
                cx, cB, cC, cdt, cA, cS = _direction(dyc[b, sl, h], xc, d["dt_c"][b, sl, h], d["B_c"][b, sl],
                                                     d["C_c"][b, sl], Af, seed, False)
                g["x_c"][b, sl, h] += cx + Df * dyc[b, sl, h]
                g["B_c"][b, sl] += cB
                g["C_c"][b, sl] += cC
                g["dt_c"][b, sl, h] += cdt
                g["A_f"][h] += cA
                g["D_f"][h] += np.sum(dyc[b, sl, h] * xc)
                if k > 0:
                    gseed[k - 1] += fS + cS
            # reverse pass over block-end states: S_k = a_k S_{k-1} + T_k
            gS = np.zeros((P, N))
            for k in range(nb - 1, -1, -1):
                sl = slice(k * Bs, (k + 1) * Bs)
                dt = d["dt_c"][b, sl, h]
                gS = gS + gseed[k] + (dst[b, k, h] if dst is not None else 0.0)
                prev = states[b, k - 1, h] if k > 0 else np.zeros((P, N))
                a = np.exp(Af * dt.sum())
                da = np.sum(gS * prev)
                g["dt_c"][b, sl, h] += Af * a * da
                g["A_f"][h] += dt.sum() * a * da
                # T_k = sum_s w_s x_s B_s^T, w_s = exp(A sum_{r>s} dt_r) dt_s
                suf = np.cumsum(dt[::-1])[::-1] - dt             # sum of dt after s in the block
                e = np.exp(Af * suf)
                w = e * dt
                x = d["x_c"][b, sl, h]
                Bb = d["B_c"][b, sl]
                gB = Bb @ gS.T                                   # (gT B_s)[p]
                g["x_c"][b, sl, h] += w[:, None] * gB
                g["B_c"][b, sl] += w[:, None] * (x @ gS)
                dw = np.sum(x * gB, axis=1)
                dsuf = Af * w * dw
                g["dt_c"][b, sl, h] += e * dw + np.concatenate([[0.0], np.cumsum(dsuf)[:-1]])
                g["A_f"][h] += float(np.sum(suf * w * dw))
                gS = a * gS
    return g


@pytest.mark.parametrize("seed,Bs,L", [(0, 4, 12), (1, 3, 9), (2, 6, 6)])
def test_planned_decomposition_matches_oracle(seed, Bs, L):
    _, d = _inputs(seed, L=L, Bs=Bs)
    y_c, y_n, st = ssd.forward(Bs, *[d[k] for k in NAMES])
    rng = np.random.default_rng(200 + seed)
    dyc, dyn, dst = rng.standard_normal(y_c.shape), rng.standard_normal(y_n.shape), rng.standard_normal(st.shape)
    want = ssd.backward(Bs, *[d[k] for k in NAMES], st, dyc, dyn, dst)
    got = planned_backward(Bs, d, st, dyc, dyn, dst)
    for k in NAMES:
        scale = max(1.0, float(np.max(np.abs(want[k]))))
        assert np.max(np.abs(got[k] - want[k])) <= 1e-10 * scale, (k, np.max(np.abs(got[k] - want[k])))
