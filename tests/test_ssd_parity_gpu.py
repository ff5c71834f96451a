"""GPU parity of the SSD (Mamba-2) form: the tcgen05 kernels through the C ABI
against the fp64 oracle (oracle/ssd.py) on the same seeded inputs, element by
element, plus the bit-exact cache properties."""

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


@pytest.fixture(scope="module", autouse=True)
def _threads(oracle_mod):
    P.oracle_threads()


def _dev(wl):
    return {k: to_device(wl.dev_bits(k), binding.BDSCAN_F32 if k in P.PARAMS or k == "init_state"
                         else binding.BDSCAN_BF16, "cuda") for k in wl.t32}


def _dims(wl, length=None):
    return binding.make_ssd_dims(wl.batch, wl.len if length is None else length, wl.block, wl.heads, wl.d_state)


def _forward(wl, t=None):
    t = t or _dev(wl)
    Bt, L, H, N = wl.batch, wl.len, wl.heads, wl.d_state
    d = _dims(wl)
    y_c = torch.empty((Bt, L, H, 64), dtype=torch.bfloat16, device="cuda")
    y_n = torch.empty_like(y_c)
    st = torch.empty((Bt, L // wl.block, H, 64, N), dtype=torch.float32, device="cuda")
    ws = torch.empty(max(1, binding.bdscan_ssd_forward_workspace_size(d)), dtype=torch.uint8, device="cuda")
    binding.ssd_forward(d, t, y_c, y_n, st, ws)
    torch.cuda.synchronize()
    assert binding.bdscan_ssd_wait_flag(1) == 0
    return t, y_c, y_n, st


def _oracle(wl, heads=None, rows=None):
    from oracle import ssd
    d = {}
    for k in NAMES:
        a = wl.f64(k)
        if heads is not None and k in P.PARAMS:
            a = a[heads]
        elif heads is not None and k.startswith(("x_", "dt_")):
            a = a[:, :, heads]
        if rows is not None and k not in P.PARAMS:
            a = a[rows]
        d[k] = np.ascontiguousarray(a)
    return ssd.forward(wl.block, *[d[k] for k in NAMES])


def _check(y_c, y_n, st, o, heads=None, rows=None):
    def pick(a):
        a = to_numpy(a)
        if rows is not None:
            a = a[rows]
        return a if heads is None else a[:, :, heads]
    P.assert_close("y_c", pick(y_c), o[0], P.FWD_TOL, P.BF16_U)
    P.assert_close("y_n", pick(y_n), o[1], P.FWD_TOL, P.BF16_U)
    P.assert_close("states", pick(st), o[2], P.FWD_TOL)


# (batch, length, block, heads, d_state): one and several blocks, both block
# sizes, both state sizes, head counts above the 8 per CTA (several head
# groups, a ragged last group)
SMALL = [(1, 256, 128, 2, 64), (2, 512, 256, 3, 128), (1, 768, 256, 9, 64), (2, 384, 128, 11, 128),
         (1, 256, 256, 1, 128)]


@pytest.mark.parametrize("cfg", SMALL)
def test_ssd_forward_matches_oracle(cfg):
    wl = SsdWorkload(*cfg, seed=1)
    _, y_c, y_n, st = _forward(wl)
    _check(y_c, y_n, st, _oracle(wl))


@pytest.mark.parametrize("cfg,heads,rows", [((8, 8192, 256, 26, 128), [0, 25], [5]),
                                            ((8, 8192, 256, 14, 64), [3, 13], [0])])
def test_ssd_full_size_sampled(cfg, heads, rows):
    """The 350M-class (26 heads of 64, state 128) and 87M-class (14 heads,
    state 64) Mamba-2 layers at training size (batch 8, 8192 tokens per
    stream, block 256), in the bench's launch configuration; the oracle runs
    two heads of one batch row (heads and batch rows are independent given
    the shared B, C)."""
    wl = SsdWorkload(*cfg, seed=0)
    _, y_c, y_n, st = _forward(wl)
    _check(y_c, y_n, st, _oracle(wl, heads=heads, rows=rows), heads=heads, rows=rows)


def test_ssd_cache_paths_are_bit_exact():
    wl = SsdWorkload(2, 1024, 256, 5, 128, seed=2, with_init=True)
    t, y_c, y_n, st = _forward(wl)
    d = _dims(wl)
    Bt, L, H, N, Bs = wl.batch, wl.len, wl.heads, wl.d_state, wl.block
    # cache build: every block-end state and the clean output, same bits
    st2 = torch.empty_like(st)
    y2 = torch.empty_like(y_c)
    ws = torch.empty(binding.bdscan_ssd_boundary_states_workspace_size(d, 1), dtype=torch.uint8, device="cuda")
    binding.ssd_boundary_states(d, t, None, y2, st2, 1, ws)
    # final state only
    fin = torch.empty((Bt, 1, H, 64, N), dtype=torch.float32, device="cuda")
    ws0 = torch.empty(binding.bdscan_ssd_boundary_states_workspace_size(d, 0), dtype=torch.uint8, device="cuda")
    binding.ssd_boundary_states(d, t, None, None, fin, 0, ws0)
    torch.cuda.synchronize()
    assert torch.equal(st2, st) and torch.equal(y2, y_c) and torch.equal(fin[:, 0], st[:, -1])
    # active block k from the cached state equals the all-block output
    da = binding.make_ssd_dims(Bt, Bs, Bs, H, N)
    for k in (0, 1, L // Bs - 1):
        sl = slice(k * Bs, (k + 1) * Bs)
        tk = {n: (v[:, sl].contiguous() if v.dim() >= 3 else v) for n, v in t.items()}
        ya = torch.empty((Bt, Bs, H, 64), dtype=torch.bfloat16, device="cuda")
        seed = st[:, k - 1].contiguous() if k > 0 else None
        binding.ssd_active_block(da, seed, tk, ya)
        torch.cuda.synchronize()
        assert torch.equal(ya, y_n[:, sl]), k
    # cache append from an initial state matches the oracle
    half = L // 2
    dh = binding.make_ssd_dims(Bt, half, Bs, H, N)
    th = {n: (v[:, half:].contiguous() if v.dim() >= 3 and n != "init_state" else v) for n, v in t.items()}
    st3 = torch.empty((Bt, half // Bs, H, 64, N), dtype=torch.float32, device="cuda")
    y3 = torch.empty((Bt, half, H, 64), dtype=torch.bfloat16, device="cuda")
    ws3 = torch.empty(binding.bdscan_ssd_boundary_states_workspace_size(dh, 1), dtype=torch.uint8, device="cuda")
    binding.ssd_boundary_states(dh, th, t["init_state"], y3, st3, 1, ws3)
    torch.cuda.synchronize()
    assert binding.bdscan_ssd_wait_flag(1) == 0
    from oracle import ssd
    ost, oy = ssd.boundary_states(Bs, *[wl.f64(k)[:, half:] for k in ("x_c", "dt_c", "B_c", "C_c")],
                                  wl.f64("A_f"), wl.f64("D_f"), init_state=wl.f64("init_state"), want_y=True)
    P.assert_close("states (append)", to_numpy(st3), ost, P.FWD_TOL)
    P.assert_close("y_c (append)", to_numpy(y3), oy, P.FWD_TOL, P.BF16_U)


def test_ssd_deterministic():
    wl = SsdWorkload(1, 512, 256, 4, 64, seed=3)
    t, y_c, y_n, st = _forward(wl)
    _, y_c2, y_n2, st2 = _forward(wl, t)
    assert torch.equal(y_c, y_c2) and torch.equal(y_n, y_n2) and torch.equal(st, st2)


def test_ssd_bounded_wait_reports_instead_of_hanging():
    """A wait that nothing completes gives up after its poll limit, sets the
    device flag and returns; the context stays usable for the next call."""
    assert binding.bdscan_ssd_wait_selftest(256) == 1
    assert binding.bdscan_ssd_wait_flag(0) == 0
    wl = SsdWorkload(1, 256, 128, 2, 64, seed=4)
    _, y_c, y_n, st = _forward(wl)
    _check(y_c, y_n, st, _oracle(wl))


@pytest.mark.parametrize("cfg", [(1, 512, 256, 3, 128), (2, 384, 128, 5, 64)])
def test_ssd_full_bidir_matches_oracle(cfg):
    """Full-sequence bidirectional SSD layer against the oracle: one noisy block
    spanning the whole sequence (seed 0) is exactly that layer."""
    from oracle import ssd
    wl = SsdWorkload(*cfg, seed=6)
    t = _dev(wl)
    d = _dims(wl)
    y = torch.empty((wl.batch, wl.len, wl.heads, 64), dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(binding.bdscan_ssd_full_bidir_workspace_size(d), dtype=torch.uint8, device="cuda")
    binding.ssd_full_bidir_forward(d, t, y, ws)
    torch.cuda.synchronize()
    assert binding.bdscan_ssd_wait_flag(1) == 0
    z = {k: np.zeros_like(wl.f64(k)) for k in ("x_c", "dt_c", "B_c", "C_c")}
    args = [z[k] if k in z else wl.f64(k) for k in NAMES]
    _, y_ref, _ = ssd.forward(wl.len, *args)
    P.assert_close("y (full bidirectional)", to_numpy(y), y_ref, P.FWD_TOL, P.BF16_U)


def test_operand_tiles_arrive_by_tma():
    """On GB300 the left-to-right scans take their x tiles and seeds through
    the tensor memory accelerator (the parity tests above then cover that
    path); right-to-left streams keep cp.async."""
    assert binding.bdscan_ssd_tma_enabled() == 1
