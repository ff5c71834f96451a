"""GPU parity of the SSD-form backward (bdscan_ssd_backward, tcgen05) against the
fp64 oracle (oracle/ssd.py::backward, pinned by finite differences and the
exact matrix-form gradients) on the same seeded inputs, every gradient at
the gradient tolerance, plus run-to-run determinism."""

import numpy as np
import pytest

import parity as P
from paper_2607_02805_gb300.inputs import SsdWorkload

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover - collected on CPU machines
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2607_02805_gb300 import binding  # noqa: E402
from paper_2607_02805_gb300.layer import to_device, to_numpy  # noqa: E402

NAMES = P.FWD_NAMES
TOKEN_N = ("B_c", "C_c", "B_f", "C_f", "B_r", "C_r")


@pytest.fixture(scope="module", autouse=True)
def _threads(oracle_mod):
    P.oracle_threads()


def _dev(wl):
    return {k: to_device(wl.dev_bits(k), binding.BDSCAN_F32 if k in P.PARAMS or k == "dstates"
                         else binding.BDSCAN_BF16, "cuda") for k in wl.t32}


def _run(wl, use_dy_c=True, use_dstates=False):
    t = _dev(wl)
    Bt, L, H, N, Bs = wl.batch, wl.len, wl.heads, wl.d_state, wl.block
    d = binding.make_ssd_dims(Bt, L, Bs, H, N)
    y_c = torch.empty((Bt, L, H, 64), dtype=torch.bfloat16, device="cuda")
    y_n = torch.empty_like(y_c)
    st = torch.empty((Bt, L // Bs, H, 64, N), dtype=torch.float32, device="cuda")
    ws = torch.empty(binding.bdscan_ssd_forward_workspace_size(d), dtype=torch.uint8, device="cuda")
    binding.ssd_forward(d, t, y_c, y_n, st, ws)
    g = {k: torch.full(v.shape, float("nan"), dtype=torch.float32 if k in P.PARAMS else torch.bfloat16, device="cuda")
         for k, v in t.items() if k in NAMES}
    wsb = torch.empty(binding.bdscan_ssd_backward_workspace_size(d), dtype=torch.uint8, device="cuda")
    binding.ssd_backward(d, t, st, t["dy_c"] if use_dy_c else None, t["dy_n"],
                         t["dstates"] if use_dstates else None, g, wsb)
    torch.cuda.synchronize()
    assert binding.bdscan_ssd_wait_flag(1) == 0
    return t, st, g, (d, wsb)


def _oracle(wl, st, use_dy_c=True, use_dstates=False, heads=None, rows=None):
    from oracle import ssd
    d = {}
    for k in NAMES + ("dy_c", "dy_n"):
        a = wl.f64(k)
        if heads is not None and k in P.PARAMS:
            a = a[heads]
        elif heads is not None and k.startswith(("x_", "dt_", "dy_")):
            a = a[:, :, heads]
        if rows is not None and k not in P.PARAMS:
            a = a[rows]
        d[k] = np.ascontiguousarray(a)
    s = to_numpy(st)
    if heads is not None:
        s = s[:, :, heads]
    if rows is not None:
        s = s[rows]
    dst = None
    if use_dstates:
        dst = wl.f64("dstates")
        if heads is not None:
            dst = dst[:, :, heads]
        if rows is not None:
            dst = dst[rows]
    return ssd.backward(wl.block, *[d[k] for k in NAMES], s, d["dy_c"] if use_dy_c else None, d["dy_n"], dst)


def _check(g, og, heads=None, rows=None, sums=True):
    for k in NAMES:
        if k in TOKEN_N and not sums:
            continue
        if rows is not None and k in P.PARAMS:  # sums over every batch row
            continue
        a = to_numpy(g[k])
        if rows is not None and k not in P.PARAMS:
            a = a[rows]
        if heads is not None:
            if k in P.PARAMS:
                a = a[heads]
            elif k.startswith(("x_", "dt_")):
                a = a[:, :, heads]
        P.assert_close("d" + k, a, og[k], P.GRAD_TOL, 0.0 if k in P.PARAMS else P.BF16_U)


# (batch, length, block, heads, d_state): one and several blocks, both block
# sizes (one and two 128-token tiles), both state sizes
SMALL = [(1, 256, 128, 2, 64), (1, 512, 256, 2, 128), (2, 768, 256, 3, 64), (2, 512, 128, 3, 128)]


@pytest.mark.parametrize("cfg", SMALL)
def test_ssd_backward_matches_oracle(cfg):
    Bt, L, Bs, H, N = cfg
    wl = SsdWorkload(Bt, L, Bs, H, N, seed=71, with_grads=True)
    _, st, g, _ = _run(wl)
    _check(g, _oracle(wl, st))


def test_ssd_backward_external_state_gradient_and_no_clean_output_gradient():
    wl = SsdWorkload(2, 512, 256, 2, 128, seed=72, with_grads=True, with_dstates=True)
    _, st, g, _ = _run(wl, use_dy_c=False, use_dstates=True)
    _check(g, _oracle(wl, st, use_dy_c=False, use_dstates=True))


def test_ssd_backward_is_deterministic():
    wl = SsdWorkload(2, 512, 256, 3, 64, seed=73, with_grads=True)
    t, st, g, (d, wsb) = _run(wl)
    first = {k: v.clone() for k, v in g.items()}
    binding.ssd_backward(d, t, st, t["dy_c"], t["dy_n"], None, g, wsb)
    torch.cuda.synchronize()
    for k in first:
        assert torch.equal(first[k], g[k]), k


def test_ssd_cp_async_path_matches_tma_bit_exact():
    """The cp.async staging (taken where the driver has no tensor-map encoder)
    gives the same bits as the TMA path, forward and backward: the arithmetic
    does not depend on how the tiles arrive."""
    wl = SsdWorkload(2, 512, 256, 3, 128, seed=74, with_grads=True)

    def both():
        t, st, g, (d, _) = _run(wl)
        y_c = torch.empty((wl.batch, wl.len, wl.heads, 64), dtype=torch.bfloat16, device="cuda")
        y_n = torch.empty_like(y_c)
        ws = torch.empty(binding.bdscan_ssd_forward_workspace_size(d), dtype=torch.uint8, device="cuda")
        binding.ssd_forward(d, t, y_c, y_n, torch.empty_like(st), ws)
        torch.cuda.synchronize()
        return st, dict(g, y_c=y_c, y_n=y_n)

    assert binding.bdscan_ssd_set_tma(1) == 1
    st_tma, out_tma = both()
    try:
        assert binding.bdscan_ssd_set_tma(0) == 0
        st_cp, out_cp = both()
    finally:
        binding.bdscan_ssd_set_tma(1)
    assert binding.bdscan_ssd_wait_flag(1) == 0
    assert torch.equal(st_tma, st_cp)
    for k in out_tma:
        assert torch.equal(out_tma[k], out_cp[k]), k


def test_bench_event_lists_match_launches():
    """bench.py times every SSD kernel with one CUDA event per launch, so its
    kernel lists must name each launch of a forward and of a backward call."""
    import importlib.util
    import os
    path = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "bench.py")
    spec = importlib.util.spec_from_file_location("bench_lists", path)
    bench = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(bench)
    wl = SsdWorkload(2, 512, 256, 3, 128, seed=75, with_grads=True)
    t = _dev(wl)
    d = binding.make_ssd_dims(wl.batch, wl.len, wl.block, wl.heads, wl.d_state)
    y_c = torch.empty((wl.batch, wl.len, wl.heads, 64), dtype=torch.bfloat16, device="cuda")
    y_n = torch.empty_like(y_c)
    st = torch.empty((wl.batch, wl.len // wl.block, wl.heads, 64, wl.d_state), dtype=torch.float32, device="cuda")
    ws = torch.empty(binding.bdscan_ssd_forward_workspace_size(d), dtype=torch.uint8, device="cuda")
    binding.ssd_forward(d, t, y_c, y_n, st, ws)
    assert binding.bdscan_last_launch_count() == len(bench.SSD_KERNELS)
    g = {k: torch.empty(v.shape, dtype=torch.float32 if k in P.PARAMS else torch.bfloat16, device="cuda")
         for k, v in t.items() if k in NAMES}
    wsb = torch.empty(binding.bdscan_ssd_backward_workspace_size(d), dtype=torch.uint8, device="cuda")
    binding.ssd_backward(d, t, st, t["dy_c"], t["dy_n"], None, g, wsb)
    assert binding.bdscan_last_launch_count() == len(bench.SSD_BWD_KERNELS)
    torch.cuda.synchronize()


@pytest.mark.parametrize("cfg,heads,rows", [
    ((8, 8192, 256, 26, 128), [0, 25], [3]),   # 350M-class layer
    ((8, 8192, 256, 14, 64), [7], [0]),        # 87M-class layer
])
def test_ssd_backward_full_size_sampled(cfg, heads, rows):
    """Training-size layers: per-token gradients on sampled heads of one batch
    row (heads are independent except in dB and dC, and dA, dD sum over every
    batch row; the small cases check those in full)."""
    Bt, L, Bs, H, N = cfg
    wl = SsdWorkload(Bt, L, Bs, H, N, seed=74, with_grads=True)
    _, st, g, _ = _run(wl)
    og = _oracle(wl, st, heads=heads, rows=rows)
    _check(g, og, heads=heads, rows=rows, sums=False)
