"""GPU parity: the CUDA library (through the C ABI) against the fp64 oracle on
the same seeded inputs, element by element, plus the bit-exact properties of
the method (cache reuse, seed indexing, determinism)."""

import numpy as np
import pytest

import parity as P
from paper_2607_02805_gb300.inputs import Workload

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():  # pragma: no cover - collected on CPU machines
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2607_02805_gb300 import binding  # noqa: E402
from paper_2607_02805_gb300.layer import Layer, to_device, to_numpy  # noqa: E402


@pytest.fixture(scope="module", autouse=True)
def _threads(oracle_mod):
    P.oracle_threads()


def _u(lay):
    return P.BF16_U if lay.out_torch == torch.bfloat16 else 0.0


def _check_forward(lay, y_c, y_n, st, sub=None):
    pick = (lambda a: a) if sub is None else (lambda a: a[:, :, sub])
    P.assert_close("y_c", pick(to_numpy(lay.y_c)), y_c, P.FWD_TOL, _u(lay))
    P.assert_close("y_n", pick(to_numpy(lay.y_n)), y_n, P.FWD_TOL, _u(lay))
    P.assert_close("states", pick(to_numpy(lay.states)), st, P.FWD_TOL)


def _check_grads(lay, g, sub=None, names=None):
    for k in names or P.FWD_NAMES:
        gpu = to_numpy(lay.g[k])
        if sub is not None:
            if k in ("A_f", "A_r", "D_f", "D_r"):
                gpu = gpu[sub]
            elif gpu.ndim == 3 and k not in ("B_c", "C_c", "B_f", "C_f", "B_r", "C_r"):
                gpu = gpu[:, :, sub]
        u = 0.0 if k in P.PARAMS else _u(lay)
        P.assert_close("d" + k, gpu, g[k], P.GRAD_TOL, u)


SMALL = [  # (Bt, L, Bs, D, N, dtype, out_dtype, seed)
    (1, 256, 16, 32, 8, "f32", None, 0),          # the tiny correctness configuration
    (2, 400, 16, 136, 16, "bf16", binding.BDSCAN_F32, 1),   # ragged last chunk and channel group
    (2, 400, 16, 136, 16, "bf16", None, 2),
    (1, 384, 4, 64, 16, "bf16", binding.BDSCAN_F32, 3),
    (1, 256, 32, 128, 16, "bf16", binding.BDSCAN_F32, 4),   # backward in 2 segments per block
    (1, 256, 64, 64, 8, "bf16", binding.BDSCAN_F32, 5),     # 4 segments, N = 8
    (2, 96, 1, 40, 16, "f32", None, 6),           # block size 1
    (1, 288, 48, 48, 16, "f32", None, 7),         # 3 segments, 2-block chunks, ragged chunk
    (3, 256, 8, 256, 8, "bf16", binding.BDSCAN_F32, 8),
    (1, 384, 128, 136, 16, "bf16", None, 9),     # 8 segments per block, one block per chunk
    (2, 256, 128, 64, 8, "f32", None, 10),
    (1, 384, 96, 64, 16, "bf16", binding.BDSCAN_F32, 14),  # 6 segments, 96-token chunks
    (2, 512, 256, 136, 16, "bf16", None, 15),    # 16 segments: checkpoints in global memory
    (1, 512, 256, 64, 8, "f32", None, 16),
]


@pytest.mark.parametrize("Bt,L,Bs,D,N,dt,od,seed", SMALL)
def test_forward_backward_parity(Bt, L, Bs, D, N, dt, od, seed):
    wl = Workload(Bt, L, Bs, D, N, dtype=dt, seed=seed, with_grads=True)
    lay = Layer(wl, out_dtype=od)
    lay.forward()
    lay.backward(use_dstates=False)
    torch.cuda.synchronize()
    y_c, y_n, st = P.oracle_forward(wl)
    _check_forward(lay, y_c, y_n, st)
    g = P.oracle_backward(wl, st)
    _check_grads(lay, g)


def test_external_state_gradient_and_no_clean_output_gradient():
    wl = Workload(2, 512, 16, 128, 16, dtype="bf16", seed=11, with_grads=True, with_dstates=True)
    lay = Layer(wl, out_dtype=binding.BDSCAN_F32)
    lay.forward()
    lay.backward(use_dy_c=False, use_dstates=True)
    torch.cuda.synchronize()
    _, _, st = P.oracle_forward(wl)
    g = P.oracle_backward(wl, st, use_dy_c=False, use_dstates=True)
    _check_grads(lay, g)


def test_backward_is_deterministic():
    wl = Workload(2, 512, 16, 256, 16, dtype="bf16", seed=12, with_grads=True)
    lay = Layer(wl)
    lay.forward()
    lay.backward(use_dstates=False)
    first = {k: v.clone() for k, v in lay.g.items()}
    lay.backward(use_dstates=False)
    torch.cuda.synchronize()
    for k in first:
        assert torch.equal(first[k], lay.g[k]), k


def test_seed_indexing_invariant_bit_exact():
    """Noisy stream = clean stream, reverse direction off: every noisy block
    continues the clean state, so y_n equals y_c bit for bit."""
    wl = Workload(2, 512, 16, 128, 16, dtype="bf16", seed=13, with_grads=False)
    for a, b_ in (("x_n", "x_c"), ("dt_f", "dt_c"), ("B_f", "B_c"), ("C_f", "C_c")):
        wl.override(a, wl.t32[b_])
    wl.override("B_r", np.zeros_like(wl.t32["B_r"]))
    wl.override("D_r", np.zeros_like(wl.t32["D_r"]))
    lay = Layer(wl)
    lay.forward()
    torch.cuda.synchronize()
    assert torch.equal(lay.y_n, lay.y_c)


def _boundary(wl, emit_all, init=None, want_y=False):
    Bt, L, Bs, D, N = wl.batch, wl.len, wl.block, wl.d_inner, wl.d_state
    dt = binding.BDSCAN_BF16 if wl.dtype == "bf16" else binding.BDSCAN_F32
    dims = binding.make_dims(Bt, L, Bs, D, N, dt)
    t = {k: to_device(wl.dev_bits(k), dt, "cuda") for k in ("x_c", "dt_c", "B_c", "C_c", "A_f", "D_f")}
    nS = (L // Bs) if emit_all else 1
    st = torch.zeros((Bt, nS, D, N), dtype=torch.float32, device="cuda")
    y = torch.zeros((Bt, L, D), dtype=t["x_c"].dtype, device="cuda") if want_y else None
    ws = torch.zeros((binding.bdscan_boundary_states_workspace_size(dims, emit_all) + 3) // 4, dtype=torch.float32,
                     device="cuda")
    binding.boundary_states(dims, t, init, y, st, emit_all, ws)
    return st, y


def _active(wl_blk, seed_states):
    Bt, Bs, D, N = wl_blk.batch, wl_blk.block, wl_blk.d_inner, wl_blk.d_state
    dt = binding.BDSCAN_BF16 if wl_blk.dtype == "bf16" else binding.BDSCAN_F32
    dims = binding.make_dims(Bt, Bs, Bs, D, N, dt)
    t = {k: to_device(wl_blk.dev_bits(k), dt, "cuda") for k in wl_blk.t32}
    y = torch.zeros((Bt, Bs, D), dtype=t["x_n"].dtype, device="cuda")
    binding.active_block(dims, seed_states.contiguous(), t, y)
    return y


def _sub_workload(wl, lo, hi):
    """A view of tokens [lo, hi) of a workload (same seeds, same values)."""
    w = object.__new__(Workload)
    w.__dict__.update(wl.__dict__)
    w.t32 = {k: (np.ascontiguousarray(v[:, lo:hi]) if v.ndim == 3 else v) for k, v in wl.t32.items()}
    w.len = hi - lo
    return w


@pytest.mark.parametrize("L,Bs", [(512, 16), (400, 16), (384, 32), (256, 4)])
def test_cache_reuse_is_bit_exact(L, Bs):
    """boundary_states over the prefix, then active_block from its final state,
    equals the last noisy block of the all-block forward bit for bit; the
    emitted boundary states equal the forward's."""
    wl = Workload(2, L, Bs, 136, 16, dtype="bf16", seed=21, with_grads=False)
    lay = Layer(wl)
    lay.forward()
    pre = _sub_workload(wl, 0, L - Bs)
    fin, _ = _boundary(pre, emit_all=False)
    allst, _ = _boundary(pre, emit_all=True)
    fin_y, y_pre = _boundary(pre, emit_all=False, want_y=True)
    blk = _sub_workload(wl, L - Bs, L)
    y = _active(blk, fin[:, 0])
    torch.cuda.synchronize()
    assert torch.equal(allst, lay.states[:, :-1])
    assert torch.equal(fin[:, 0], lay.states[:, -2])
    assert torch.equal(fin_y, fin)
    assert torch.equal(y_pre, lay.y_c[:, : L - Bs])
    assert torch.equal(y, lay.y_n[:, L - Bs:])


def test_cache_append_matches_single_scan():
    """Appending to the cache (init_state = previous final state) equals one
    scan over the concatenation; bit exact when the first part is a whole
    number of time chunks."""
    Bs = 16
    tc = binding.bdscan_chunk_tokens(Bs)
    wl = Workload(1, 3 * tc, Bs, 128, 16, dtype="bf16", seed=22, with_grads=False)
    full, _ = _boundary(wl, emit_all=False)
    a, _ = _boundary(_sub_workload(wl, 0, tc), emit_all=False)
    b_, _ = _boundary(_sub_workload(wl, tc, 3 * tc), emit_all=False, init=a[:, 0].contiguous())
    torch.cuda.synchronize()
    assert torch.equal(full, b_)
    # and against the oracle, appended from an oracle state
    import oracle
    d = P.slice_channels(wl, None)
    ofin, _ = oracle.boundary_states(Bs, d["x_c"], d["dt_c"], d["B_c"], d["C_c"], d["A_f"], d["D_f"], emit_all=False)
    P.assert_close("appended state", to_numpy(b_), ofin, P.FWD_TOL)


def test_zero_size_calls_are_noops():
    dims = binding.make_dims(0, 64, 16, 32, 16, binding.BDSCAN_BF16)
    assert binding.bdscan_forward_workspace_size(dims) >= 0
    wl = Workload(1, 16, 16, 32, 16, dtype="bf16", seed=1, with_grads=False)
    st, _ = _boundary(_sub_workload(wl, 0, 0), emit_all=False)
    torch.cuda.synchronize()
    assert torch.count_nonzero(st) == 0


# ---------------------------------------------------------------------------
# full-sequence bidirectional layer (the DiffuMamba comparator)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("Bt,L,Bs,D,N,dt,od,seed", [
    (2, 512, 16, 136, 16, "bf16", None, 31),               # ragged channel group
    (1, 400, 16, 64, 8, "f32", None, 32),                  # ragged last chunk, N = 8
    (2, 384, 32, 128, 16, "bf16", binding.BDSCAN_F32, 33),  # 32-token chunking blocks, fp32 output
    (1, 256, 4, 64, 16, "bf16", None, 34),                 # tiled 4-token chunking blocks
])
def test_full_bidir_matches_oracle(Bt, L, Bs, D, N, dt, od, seed):
    """Forward and reverse scans over the whole sequence: the oracle's
    all-block forward with one block spanning the sequence (its noisy output
    is exactly that layer; the block size of the call only sets the chunking)."""
    import oracle
    wl = Workload(Bt, L, Bs, D, N, dtype=dt, seed=seed, with_grads=False, parts=("noisy",))
    code = binding.BDSCAN_F32 if dt == "f32" else binding.BDSCAN_BF16
    dims = binding.make_dims(Bt, L, Bs, D, N, code, od)
    t = {k: to_device(wl.dev_bits(k), code, "cuda") for k in wl.t32}
    out_t = torch.float32 if (dt == "f32" or od == binding.BDSCAN_F32) else torch.bfloat16
    y = torch.full((Bt, L, D), float("nan"), dtype=out_t, device="cuda")
    nbytes = binding.bdscan_full_bidir_workspace_size(dims)
    ws = torch.empty((nbytes + 3) // 4, dtype=torch.float32, device="cuda")
    binding.full_bidir_forward(dims, t, y, ws)
    torch.cuda.synchronize()
    d = P.slice_channels(wl, None)
    zeros = np.zeros_like(d["x_n"])
    zrow = np.zeros_like(d["B_f"])
    _, y_n, _ = oracle.forward(L, zeros, zeros, zrow, zrow, d["x_n"], d["dt_f"], d["B_f"], d["C_f"], d["dt_r"],
                               d["B_r"], d["C_r"], d["A_f"], d["D_f"], d["A_r"], d["D_r"])
    P.assert_close("y", to_numpy(y), y_n, P.FWD_TOL, P.BF16_U if out_t == torch.bfloat16 else 0.0)


# ---------------------------------------------------------------------------
# full-size configurations, in the launch configuration the benchmark times
# ---------------------------------------------------------------------------
def _batch_row(wl, b):
    w = object.__new__(Workload)
    w.__dict__.update(wl.__dict__)
    w.t32 = {k: (np.ascontiguousarray(v[b:b + 1]) if v.ndim >= 3 else v) for k, v in wl.t32.items()}
    w.batch = 1
    return w


def _full_size_check(Bt, L, Bs, D, N, seed, sub, sums_row):
    wl = Workload(Bt, L, Bs, D, N, dtype="bf16", seed=seed, with_grads=True)
    lay = Layer(wl)
    lay.forward()
    lay.backward(use_dstates=False)
    torch.cuda.synchronize()
    # per-channel outputs and parameter gradients on a channel sample
    y_c, y_n, st = P.oracle_forward(wl, sub=sub)
    _check_forward(lay, y_c, y_n, st, sub=sub)
    g = P.oracle_backward(wl, st, sub=sub)
    _check_grads(lay, g, sub=sub, names=[k for k in P.FWD_NAMES if k not in ("B_c", "C_c", "B_f", "C_f", "B_r", "C_r")])
    if sums_row is not None:
        # the sums over channels (dB, dC) of one batch row, all channels
        row = _batch_row(wl, sums_row)
        _, _, st1 = P.oracle_forward(row)
        g1 = P.oracle_backward(row, st1)
        for k in ("B_c", "C_c", "B_f", "C_f", "B_r", "C_r"):
            P.assert_close("d" + k, to_numpy(lay.g[k])[sums_row:sums_row + 1], g1[k], P.GRAD_TOL, _u(lay))


def test_config_87m_layer_full_size():
    """batch 8, 2048 tokens per stream, block 16, d_inner 1536, d_state 16, bf16:
    every channel of one 128-channel group (one CTA's channels: all warps and
    lanes) plus the edges of others, and dB, dC over all channels of a batch row."""
    sub = sorted({0, 1, 2, 31, 127, 128, 129, 700, 1023, 1024, 1534, 1535} | set(range(384, 512)))
    _full_size_check(8, 2048, 16, 1536, 16, 0, sub, sums_row=3)


@pytest.mark.parametrize("Bs", [4, 8, 16, 32, 64])
def test_config_350m_block_sweep_full_size(Bs):
    """batch 8, 2048 tokens, d_inner 2048, d_state 16, bf16, block size sweep."""
    sub = sorted({0, 5, 255, 256, 1337, 2047} | set(range(1536, 1664)))  # edges and one 128-channel group
    _full_size_check(8, 2048, Bs, 2048, 16, 1, sub, sums_row={4: 0, 8: 2, 16: 5, 32: 6, 64: 7}[Bs])


def _long_context(L, Bs, calls, seed):
    D, N = 2048, 16
    wl = Workload(1, L, Bs, D, N, dtype="bf16", seed=seed, with_grads=False, parts=("clean",))
    fin, _ = _boundary(wl, emit_all=False)
    sub = [0, 77, 1024, 2047]
    import oracle
    d = P.slice_channels(wl, sub)
    ofin, _ = oracle.boundary_states(Bs, d["x_c"], d["dt_c"], d["B_c"], d["C_c"], d["A_f"], d["D_f"], emit_all=False)
    P.assert_close("final state", to_numpy(fin)[:, :, sub], ofin, P.FWD_TOL)
    for j in range(calls):
        blk = Workload(1, Bs, Bs, D, N, dtype="bf16", seed=seed, with_grads=False, parts=("noisy",), part=j + 1)
        y = _active(blk, fin[:, 0])
        db = P.slice_channels(blk, sub)
        oy = oracle.active_block(ofin[:, 0], db["x_n"], db["dt_f"], db["B_f"], db["C_f"], db["dt_r"], db["B_r"],
                                 db["C_r"], db["A_f"], db["D_f"], db["A_r"], db["D_r"])
        P.assert_close(f"active block {j}", to_numpy(y)[:, :, sub], oy, P.FWD_TOL, P.BF16_U)
    return wl, fin


def test_config_long_context_65k():
    """Cache build over a 65,536-token prefix (d_inner 2048, block 32), then one
    active block; the active block equals full recomputation bit for bit."""
    L, Bs = 65536, 32
    wl, fin = _long_context(L, Bs, 1, seed=4)
    # full recomputation: the all-block forward over prefix + one block whose
    # last noisy block is the active block
    blk = Workload(1, Bs, Bs, 2048, 16, dtype="bf16", seed=4, with_grads=False, parts=("noisy",), part=1)
    full = object.__new__(Workload)
    full.__dict__.update(wl.__dict__)
    full.len = L + Bs
    full.t32 = dict(wl.t32)
    for k in ("x_c", "dt_c", "B_c", "C_c"):
        full.t32[k] = np.concatenate([wl.t32[k], wl.t32[k][:, :Bs]], axis=1)
    for k in ("x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r"):
        filler = np.zeros((1, L) + blk.t32[k].shape[2:], dtype=np.float32)
        full.t32[k] = np.concatenate([filler, blk.t32[k]], axis=1)
    for k in ("A_r", "D_r"):
        full.t32[k] = blk.t32[k]
    lay = Layer(full)
    lay.forward()
    y = _active(blk, fin[:, 0])
    torch.cuda.synchronize()
    assert torch.equal(lay.states[:, -2], fin[:, 0])
    assert torch.equal(y, lay.y_n[:, L:])


def test_config_very_long_context_262k():
    """Cache build over 262,144 tokens (block 16), then 16 active-block calls
    reusing the same read-only cached state."""
    _long_context(262144, 16, 16, seed=5)


# ---------------------------------------------------------------------------
# the forward side at the paper's block sizes (128 and 256 tokens)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("Bt,L,Bs,D,N,dt,seed", [
    (2, 512, 128, 136, 16, "bf16", 41),   # one block per chunk, ragged channel group
    (1, 768, 256, 64, 8, "f32", 42),
    (1, 512, 256, 64, 32, "bf16", 43),    # with state groups
])
def test_long_block_forward_parity_and_cache(Bt, L, Bs, D, N, dt, seed):
    """All-block forward against the oracle; cache build and the cached
    active block reproduce it bit for bit."""
    wl = Workload(Bt, L, Bs, D, N, dtype=dt, seed=seed, with_grads=False)
    lay = Layer(wl)
    lay.forward()
    torch.cuda.synchronize()
    y_c, y_n, st = P.oracle_forward(wl)
    _check_forward(lay, y_c, y_n, st)
    pre = _sub_workload(wl, 0, L - Bs)
    fin, _ = _boundary(pre, emit_all=False)
    allst, y_pre = _boundary(pre, emit_all=True, want_y=True)
    y = _active(_sub_workload(wl, L - Bs, L), fin[:, 0])
    torch.cuda.synchronize()
    assert torch.equal(allst, lay.states[:, :-1])
    assert torch.equal(fin[:, 0], lay.states[:, -2])
    assert torch.equal(y_pre, lay.y_c[:, : L - Bs])
    assert torch.equal(y, lay.y_n[:, L - Bs:])
