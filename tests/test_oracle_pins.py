"""Pins of the fp64 oracle against facts that do not come from the oracle.

Each check names what fixes it: the explicit matrix form of the scan
(independent of any recurrence), linearity, closed forms for block size 1,
dt = 0 and x = 0, the invariants stated for the method (a single block is a
full-sequence reverse scan; the seed of block k is the clean state after
block k-1; the cache reused by an active block equals full recomputation),
central finite differences, and a hand-worked example.
"""

import json
import os

import numpy as np
import pytest

import bruteforce
from paper_2607_02805_gb300.inputs import Workload

FWD = ("x_c", "dt_c", "B_c", "C_c", "x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r",
       "A_f", "D_f", "A_r", "D_r")
NOISY = ("x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r", "A_f", "D_f", "A_r", "D_r")
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def wdict(w):
    return {k: w.f64(k) for k in w.t32}


def ofwd(oracle, block, d):
    return oracle.forward(block, *[d[k] for k in FWD])


def relmax(a, b):
    den = max(np.max(np.abs(b)), 1e-300)
    return float(np.max(np.abs(a - b)) / den)


CASES = [  # (Bt, L, Bs, D, N, seed)
    (2, 12, 4, 3, 4, 0),
    (1, 8, 8, 2, 3, 1),   # a single block
    (1, 6, 1, 2, 2, 2),   # block size 1
    (2, 9, 3, 2, 5, 3),
]


@pytest.mark.parametrize("Bt,L,Bs,D,N,seed", CASES)
def test_forward_equals_matrix_form(oracle_mod, Bt, L, Bs, D, N, seed):
    """Eq. mamba-scan-background unrolled: y = M x with M built from explicit
    sums of dt; boundary states per eq. boundary-state; eq. partial-reverse."""
    w = Workload(Bt, L, Bs, D, N, dtype="f32", seed=seed, with_grads=False)
    d = wdict(w)
    y_c, y_n, st = ofwd(oracle_mod, Bs, d)
    by_c, by_n, bst = bruteforce.forward(Bs, d)
    assert relmax(y_c, by_c) < 1e-12
    assert relmax(st, bst) < 1e-12
    assert relmax(y_n, by_n) < 1e-12


def test_dx_is_transpose_of_linear_map(oracle_mod):
    """The outputs are linear in (x_c, x_n), so the exact gradient with respect
    to x is J^T applied to (dy_c, dy_n, dstates). This covers the path from a
    noisy block's loss through its cached seed into the clean prefix
    (eq. prefix-cache-gradient)."""
    Bt, L, Bs, D, N = 1, 8, 2, 2, 3
    w = Workload(Bt, L, Bs, D, N, dtype="f32", seed=5, with_grads=True, with_dstates=True)
    d = wdict(w)
    J = bruteforce.linear_map_x(Bs, d)
    y_c, y_n, st = ofwd(oracle_mod, Bs, d)
    g = oracle_mod.backward(Bs, *[d[k] for k in FWD], st, d["dy_c"], d["dy_n"], d["dstates"])
    up = np.concatenate([d["dy_c"].ravel(), d["dy_n"].ravel(), d["dstates"].ravel()])
    ref = J.T @ up
    nx = Bt * L * D
    assert relmax(g["x_c"].ravel(), ref[:nx]) < 1e-12
    assert relmax(g["x_n"].ravel(), ref[nx:]) < 1e-12


def _loss(oracle, Bs, d):
    y_c, y_n, st = ofwd(oracle, Bs, d)
    return float(np.sum(d["dy_c"] * y_c) + np.sum(d["dy_n"] * y_n) + np.sum(d["dstates"] * st))


@pytest.mark.parametrize("Bt,L,Bs,D,N,seed", [(2, 12, 4, 3, 4, 7), (1, 10, 5, 2, 2, 8), (1, 6, 1, 2, 3, 9)])
def test_backward_matches_central_differences(oracle_mod, Bt, L, Bs, D, N, seed):
    """<grad, v> against (Loss(p + eps v) - Loss(p - eps v)) / (2 eps) for a
    random direction v in every input, Loss = <dy_c,y_c>+<dy_n,y_n>+<dS,S>."""
    w = Workload(Bt, L, Bs, D, N, dtype="f32", seed=seed, with_grads=True, with_dstates=True)
    d = wdict(w)
    _, _, st = ofwd(oracle_mod, Bs, d)
    g = oracle_mod.backward(Bs, *[d[k] for k in FWD], st, d["dy_c"], d["dy_n"], d["dstates"])
    rng = np.random.default_rng(seed + 100)
    eps = 1e-6
    for name in FWD:
        v = rng.standard_normal(d[name].shape)
        dp, dm = dict(d), dict(d)
        dp[name] = d[name] + eps * v
        dm[name] = d[name] - eps * v
        fd = (_loss(oracle_mod, Bs, dp) - _loss(oracle_mod, Bs, dm)) / (2 * eps)
        an = float(np.sum(g[name] * v))
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (name, fd, an)


def test_backward_elementwise_central_differences(oracle_mod):
    """Single elements of every gradient, including the seed path."""
    Bt, L, Bs, D, N = 1, 8, 4, 2, 2
    w = Workload(Bt, L, Bs, D, N, dtype="f32", seed=11, with_grads=True, with_dstates=True)
    d = wdict(w)
    _, _, st = ofwd(oracle_mod, Bs, d)
    g = oracle_mod.backward(Bs, *[d[k] for k in FWD], st, d["dy_c"], d["dy_n"], d["dstates"])
    rng = np.random.default_rng(3)
    eps = 1e-6
    for name in FWD:
        flat = d[name].ravel()
        for idx in rng.choice(flat.size, size=min(4, flat.size), replace=False):
            dp, dm = dict(d), dict(d)
            a, b = flat.copy(), flat.copy()
            a[idx] += eps
            b[idx] -= eps
            dp[name] = a.reshape(d[name].shape)
            dm[name] = b.reshape(d[name].shape)
            fd = (_loss(oracle_mod, Bs, dp) - _loss(oracle_mod, Bs, dm)) / (2 * eps)
            an = g[name].ravel()[idx]
            assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (name, idx, fd, an)


def test_single_block_is_full_sequence_reverse(oracle_mod):
    """With one block covering the whole stream, the block-local reverse scan is
    the full-sequence reverse scan of a fully bidirectional denoiser (Sec. 4,
    the DiffuMamba comparison), and the seeded forward scan of block 0 is a
    plain causal scan from zero."""
    Bt, L, D, N = 2, 16, 3, 4
    w = Workload(Bt, L, L, D, N, dtype="f32", seed=21, with_grads=False)
    d = wdict(w)
    _, y_n, _ = ofwd(oracle_mod, L, d)
    # forward direction: the causal scan of the noisy tokens from zero
    _, y_f = oracle_mod.boundary_states(L, d["x_n"], d["dt_f"], d["B_f"], d["C_f"], d["A_f"], d["D_f"],
                                        emit_all=True, want_y=True)
    # reverse direction: a causal scan of the time-reversed tokens, reversed back
    rev = lambda a: np.ascontiguousarray(a[:, ::-1])
    _, y_r = oracle_mod.boundary_states(L, rev(d["x_n"]), rev(d["dt_r"]), rev(d["B_r"]), rev(d["C_r"]),
                                        d["A_r"], d["D_r"], emit_all=True, want_y=True)
    assert relmax(y_n, y_f + rev(y_r)) < 1e-13
    # and both against the brute-force full-window matrices
    _, by_n, _ = bruteforce.forward(L, d)
    assert relmax(y_n, by_n) < 1e-12


@pytest.mark.parametrize("L,Bs", [(32, 4), (48, 16), (20, 5)])
def test_caching_is_exact(oracle_mod, L, Bs):
    """Active-block outputs from the cached boundary state equal full
    recomputation bit for bit (the cache stays valid because the reverse scan
    is local to the block, Sec. 4)."""
    Bt, D, N = 2, 3, 4
    w = Workload(Bt, L, Bs, D, N, dtype="f32", seed=31, with_grads=False)
    d = wdict(w)
    _, y_n, st = ofwd(oracle_mod, Bs, d)
    pre = {k: (np.ascontiguousarray(d[k][:, : L - Bs]) if d[k].ndim == 3 else d[k]) for k in d}
    fin, _ = oracle_mod.boundary_states(Bs, pre["x_c"], pre["dt_c"], pre["B_c"], pre["C_c"], d["A_f"],
                                        d["D_f"], emit_all=False)
    allst, _ = oracle_mod.boundary_states(Bs, pre["x_c"], pre["dt_c"], pre["B_c"], pre["C_c"], d["A_f"],
                                          d["D_f"], emit_all=True)
    assert np.array_equal(fin[:, 0], st[:, -2])
    assert np.array_equal(allst, st[:, :-1])
    blk = {k: np.ascontiguousarray(d[k][:, L - Bs:]) for k in NOISY if d[k].ndim == 3}
    yb = oracle_mod.active_block(fin[:, 0], blk["x_n"], blk["dt_f"], blk["B_f"], blk["C_f"], blk["dt_r"],
                                 blk["B_r"], blk["C_r"], d["A_f"], d["D_f"], d["A_r"], d["D_r"])
    assert np.array_equal(yb, y_n[:, L - Bs:])


def test_cache_append_is_exact(oracle_mod):
    """Appending a finalised block to the cache (a clean pass continued from
    the cached state, Sec. 3 cache interface) equals scanning the longer
    prefix from scratch."""
    Bt, L, Bs, D, N = 1, 24, 4, 3, 4
    w = Workload(Bt, L, Bs, D, N, dtype="f32", seed=41, with_grads=False)
    d = wdict(w)
    full, _ = oracle_mod.boundary_states(Bs, d["x_c"], d["dt_c"], d["B_c"], d["C_c"], d["A_f"], d["D_f"],
                                         emit_all=False)
    cut = 16
    sl = lambda a, lo, hi: np.ascontiguousarray(a[:, lo:hi])
    first, _ = oracle_mod.boundary_states(Bs, *[sl(d[k], 0, cut) for k in ("x_c", "dt_c", "B_c", "C_c")],
                                          d["A_f"], d["D_f"], emit_all=False)
    second, _ = oracle_mod.boundary_states(Bs, *[sl(d[k], cut, L) for k in ("x_c", "dt_c", "B_c", "C_c")],
                                           d["A_f"], d["D_f"], init_state=first[:, 0], emit_all=False)
    assert np.array_equal(second, full)


def test_seed_indexing_invariant(oracle_mod):
    """Noisy stream = clean stream with the reverse direction switched off
    (B_r = 0, D_r = 0): each block continues from the state after the previous
    block, so y_n equals y_c exactly. Seeding block k from states[k] instead
    of states[k-1] (an off-by-one) breaks it by O(1)."""
    Bt, L, Bs, D, N = 2, 24, 4, 3, 4
    w = Workload(Bt, L, Bs, D, N, dtype="f32", seed=51, with_grads=False)
    d = wdict(w)
    d["x_n"], d["dt_f"], d["B_f"], d["C_f"] = d["x_c"], d["dt_c"], d["B_c"], d["C_c"]
    d["B_r"] = np.zeros_like(d["B_r"])
    d["D_r"] = np.zeros_like(d["D_r"])
    y_c, y_n, st = ofwd(oracle_mod, Bs, d)
    assert np.array_equal(y_n, y_c)
    # the invariant is sensitive to a shifted seed
    k = 3
    blk = {n: np.ascontiguousarray(d[n][:, k * Bs:(k + 1) * Bs]) for n in NOISY if d[n].ndim == 3}
    wrong = oracle_mod.active_block(st[:, k], blk["x_n"], blk["dt_f"], blk["B_f"], blk["C_f"], blk["dt_r"],
                                    blk["B_r"], blk["C_r"], d["A_f"], d["D_f"], d["A_r"], d["D_r"])
    assert relmax(wrong, y_c[:, k * Bs:(k + 1) * Bs]) > 1e-2


def test_block_size_one_closed_form(oracle_mod):
    """Bs = 1: the reverse scan sees one token, y_rev_t = (C_r,t . B_r,t) dt_r,t x_t
    + D_r x_t, and the forward scan is one step from the previous state."""
    Bt, L, D, N = 2, 7, 3, 4
    w = Workload(Bt, L, 1, D, N, dtype="f32", seed=61, with_grads=False)
    d = wdict(w)
    _, y_n, st = ofwd(oracle_mod, 1, d)
    x, Af, Ar = d["x_n"], d["A_f"], d["A_r"]
    for b in range(Bt):
        for t in range(L):
            for c in range(D):
                prev = st[b, t - 1, c] if t > 0 else np.zeros(N)
                a = np.exp(d["dt_f"][b, t, c] * Af[c])
                hf = a * prev + d["dt_f"][b, t, c] * d["B_f"][b, t] * x[b, t, c]
                yf = d["C_f"][b, t] @ hf + d["D_f"][c] * x[b, t, c]
                yr = (d["C_r"][b, t] @ d["B_r"][b, t]) * d["dt_r"][b, t, c] * x[b, t, c] + d["D_r"][c] * x[b, t, c]
                assert abs(y_n[b, t, c] - (yf + yr)) <= 1e-13 * max(1.0, abs(yf + yr))


def test_zero_step_size(oracle_mod):
    """dt = 0: every decay is exp(0) = 1 and no input enters the state, so the
    clean state stays at its initial value and y = C.h0 + D x."""
    Bt, L, Bs, D, N = 1, 12, 4, 2, 3
    w = Workload(Bt, L, Bs, D, N, dtype="f32", seed=71, with_grads=False, with_init=True)
    d = wdict(w)
    for k in ("dt_c", "dt_f", "dt_r"):
        d[k] = np.zeros_like(d[k])
    y_c, y_n, st = ofwd(oracle_mod, Bs, d)
    assert np.array_equal(st, np.zeros_like(st))
    assert np.allclose(y_c, d["D_f"] * d["x_c"], rtol=0, atol=1e-15)
    assert np.allclose(y_n, (d["D_f"] + d["D_r"]) * d["x_n"], rtol=0, atol=1e-15)
    h0 = d["init_state"]
    fin, y = oracle_mod.boundary_states(Bs, d["x_c"], d["dt_c"], d["B_c"], d["C_c"], d["A_f"], d["D_f"],
                                        init_state=h0, emit_all=False, want_y=True)
    assert np.array_equal(fin[:, 0], h0)
    ref = np.einsum("bln,bdn->bld", d["C_c"], h0) + d["D_f"] * d["x_c"]
    assert relmax(y, ref) < 1e-14


def test_zero_input_is_seed_decay(oracle_mod):
    """x_n = 0: the noisy output is the cached seed decayed through the block,
    y_t = sum_n C_f,t[n] exp(A_f[n] sum_{r=t0..t} dt_f,r) seed[n]."""
    Bt, L, Bs, D, N = 1, 16, 8, 2, 3
    w = Workload(Bt, L, Bs, D, N, dtype="f32", seed=81, with_grads=False)
    d = wdict(w)
    d["x_n"] = np.zeros_like(d["x_n"])
    _, y_n, st = ofwd(oracle_mod, Bs, d)
    for c in range(D):
        cum = 0.0
        for t in range(Bs, 2 * Bs):
            cum += d["dt_f"][0, t, c]
            ref = d["C_f"][0, t] @ (np.exp(d["A_f"][c] * cum) * st[0, 0, c])
            assert abs(y_n[0, t, c] - ref) <= 1e-14 * max(1.0, abs(ref))
    assert np.array_equal(y_n[:, :Bs], np.zeros_like(y_n[:, :Bs]))


def test_hand_worked_example(oracle_mod):
    """A 4-token example worked by hand from the equations (tests/golden)."""
    with open(os.path.join(GOLDEN, "hand_worked_L4.json")) as f:
        g = json.load(f)
    d = {k: np.array(v, dtype=np.float64) for k, v in g["inputs"].items()}
    y_c, y_n, st = ofwd(oracle_mod, g["block"], d)
    assert np.allclose(y_c, np.array(g["expected"]["y_c"]), rtol=1e-14, atol=1e-14)
    assert np.allclose(y_n, np.array(g["expected"]["y_n"]), rtol=1e-14, atol=1e-14)
    assert np.allclose(st, np.array(g["expected"]["states"]), rtol=1e-14, atol=1e-14)


def test_thread_count_does_not_change_results(oracle_mod):
    Bt, L, Bs, D, N = 3, 32, 8, 5, 4
    w = Workload(Bt, L, Bs, D, N, dtype="bf16", seed=91, with_grads=True, with_dstates=True)
    d = wdict(w)
    outs = []
    for th in (1, 4):
        oracle_mod.set_threads(th)
        y_c, y_n, st = ofwd(oracle_mod, Bs, d)
        g = oracle_mod.backward(Bs, *[d[k] for k in FWD], st, d["dy_c"], d["dy_n"], d["dstates"])
        outs.append((y_c, y_n, st, g))
    oracle_mod.set_threads(1)
    for a, b in zip(outs[0][:3], outs[1][:3]):
        assert np.array_equal(a, b)
    for k in FWD:
        assert np.array_equal(outs[0][3][k], outs[1][3][k])


def test_rejects_ragged_length(oracle_mod):
    w = Workload(1, 10, 4, 2, 2, dtype="f32", seed=1, with_grads=False)
    d = wdict(w)
    with pytest.raises(ValueError):
        ofwd(oracle_mod, 4, d)
